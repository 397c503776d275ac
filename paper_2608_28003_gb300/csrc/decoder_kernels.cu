// Supporting kernels of the Gemma-3-1B-shaped decoder: embedding + RMSNorm, residual + sandwich
// RMSNorms, QK-norm + RoPE + KV-cache write, and causal (sliding-window) GQA attention.
// bf16 activations between kernels, an fp32 residual stream, fp32 arithmetic inside.
#include <cmath>

#include "decoder_kernels.cuh"

namespace w8a8 {

namespace {

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}

// Sum over the block (blockDim.x a multiple of 32, at most 1024); every thread gets the result.
__device__ float block_sum(float v, float* red) {
  v = warp_sum(v);
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  float s = 0.0f;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s += red[i];
  return s;
}

// Maximum over the block; every thread gets the result.
__device__ float block_max(float v, float* red) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  __syncthreads();
  if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = v;
  __syncthreads();
  float s = 0.0f;
  for (int i = 0; i < (int)(blockDim.x >> 5); ++i) s = fmaxf(s, red[i]);
  return s;
}

constexpr int kRowThreads = 256;
constexpr int kRowVec = 2;  // 8-element vectors per thread: H <= 4096

__device__ __forceinline__ void unpack8(const uint4& w, float (&x)[8]) {
  x[0] = bf16_lo(w.x); x[1] = bf16_hi(w.x); x[2] = bf16_lo(w.y); x[3] = bf16_hi(w.y);
  x[4] = bf16_lo(w.z); x[5] = bf16_hi(w.z); x[6] = bf16_lo(w.w); x[7] = bf16_hi(w.w);
}

__device__ __forceinline__ uint4 pack8(const float (&x)[8]) {
  uint4 w;
  w.x = (uint32_t)f32_to_bf16_bits(x[0]) | ((uint32_t)f32_to_bf16_bits(x[1]) << 16);
  w.y = (uint32_t)f32_to_bf16_bits(x[2]) | ((uint32_t)f32_to_bf16_bits(x[3]) << 16);
  w.z = (uint32_t)f32_to_bf16_bits(x[4]) | ((uint32_t)f32_to_bf16_bits(x[5]) << 16);
  w.w = (uint32_t)f32_to_bf16_bits(x[6]) | ((uint32_t)f32_to_bf16_bits(x[7]) << 16);
  return w;
}

// The next linear's per-token quantiser (K1, Eq. xhat-lmhead / stx / xint8) on the row this block
// has just produced, fused here because the block holds the whole row: x_hat = fl(x * inv_delta),
// m = max |x_hat|, s_x = fl(m / 127), codes = clamp(rint(fl(x_hat * fl(127 / m))), -127, 127) written
// as fp16 (the tensor-core GEMM's operand).  x: this thread's vectors of the row, already rounded to
// bf16 (the values the stand-alone K1 would read); the arithmetic is the stand-alone K1's, so the
// codes and s_x are bit-identical to it.
struct RowQuant {
  const float* inv_delta;  // [H]; null: no codes
  uint16_t* codes;         // [M, H] fp16
  float* s_x;              // [M]
  int* qsum;               // [M] nullable: sum_k |q_tk| (the tensor-core GEMM's exactness certificate)
};
__device__ __forceinline__ void row_quantize(const RowQuant& q, int row, int H, const float (&x)[kRowVec][8],
                                             float* red) {
  const int nv = H >> 3;
  float xh[kRowVec][8];
  float amax = 0.0f;
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        xh[v][e] = __fmul_rn(x[v][e], q.inv_delta[vi * 8 + e]);
        amax = fmaxf(amax, fabsf(xh[v][e]));
      }
    }
  }
  const float m = block_max(amax, red);
  const float r = m > 0.0f ? __fdiv_rn(127.0f, m) : 0.0f;
  if (threadIdx.x == 0) q.s_x[row] = __fdiv_rn(m, 127.0f);
#pragma unroll
  int qs = 0;
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
      uint32_t h[4];
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        const int q0 = max(-127, min(127, __float2int_rn(__fmul_rn(xh[v][2 * e], r))));
        const int q1 = max(-127, min(127, __float2int_rn(__fmul_rn(xh[v][2 * e + 1], r))));
        qs += abs(q0) + abs(q1);
        h[e] = (uint32_t)int_to_f16_bits(q0) | ((uint32_t)int_to_f16_bits(q1) << 16);
      }
      reinterpret_cast<uint4*>(q.codes + (size_t)row * H)[vi] = make_uint4(h[0], h[1], h[2], h[3]);
    }
  }
  if (q.qsum) {  // integer sum over the block (exact in any order)
    __shared__ int qred[kRowThreads / 32];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) qs += __shfl_xor_sync(0xffffffffu, qs, o);
    if ((threadIdx.x & 31) == 0) qred[threadIdx.x >> 5] = qs;
    __syncthreads();
    if (threadIdx.x == 0) {
      int t = 0;
#pragma unroll
      for (int w = 0; w < kRowThreads / 32; ++w) t += qred[w];
      q.qsum[row] = t;
    }
  }
}

__device__ __forceinline__ void round8_bf16(const float (&x)[8], float (&b)[8]) {
#pragma unroll
  for (int e = 0; e < 8; ++e) b[e] = bf16_bits_to_f32(f32_to_bf16_bits(x[e]));
}

__global__ void __launch_bounds__(kRowThreads) embed_norm_kernel(const int32_t* __restrict__ tokens, int vocab,
                                                                 const uint16_t* __restrict__ embed, int H, float scale,
                                                                 const float* __restrict__ w, float eps,
                                                                 float* __restrict__ r, uint16_t* __restrict__ a,
                                                                 const RowQuant rq) {
  pdl_trigger();
  pdl_wait();
  __shared__ float red[32];
  const int row = blockIdx.x;
  int tok = tokens[row];
  if (tok < 0 || tok >= vocab) tok = 0;  // an invalid id reads row 0 instead of faulting
  const int nv = H >> 3;
  const uint4* src = reinterpret_cast<const uint4*>(embed + (size_t)tok * H);
  float x[kRowVec][8];
  float ss = 0.0f;
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
      unpack8(src[vi], x[v]);
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        x[v][e] *= scale;
        ss += x[v][e] * x[v][e];
      }
    }
  }
  const float inv = 1.0f / sqrtf(block_sum(ss, red) / (float)H + eps);
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
      float4* rp = reinterpret_cast<float4*>(r + (size_t)row * H + vi * 8);
      rp[0] = make_float4(x[v][0], x[v][1], x[v][2], x[v][3]);
      rp[1] = make_float4(x[v][4], x[v][5], x[v][6], x[v][7]);
      float y[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) y[e] = x[v][e] * inv * w[vi * 8 + e];
      reinterpret_cast<uint4*>(a + (size_t)row * H)[vi] = pack8(y);
      if (rq.inv_delta) round8_bf16(y, x[v]);  // x now holds the bf16 row
    }
  }
  if (rq.inv_delta) row_quantize(rq, row, H, x, red);
}

__global__ void __launch_bounds__(kRowThreads) residual_norm_kernel(const uint16_t* __restrict__ y, int H,
                                                                    const float* __restrict__ w_post,
                                                                    const float* __restrict__ w_next, float eps,
                                                                    float* __restrict__ r, uint16_t* __restrict__ a,
                                                                    const RowQuant rq) {
  pdl_trigger();
  __shared__ float red[32];
  const int row = blockIdx.x;
  const int nv = H >> 3;
  // the norm weights are constants: read them before the preceding kernel has finished
  float wp[kRowVec][8], wn[kRowVec][8];
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
      const float4* p0 = reinterpret_cast<const float4*>(w_post + vi * 8);
      const float4* p1 = reinterpret_cast<const float4*>(w_next + vi * 8);
      const float4 a0 = p0[0], a1 = p0[1], b0 = p1[0], b1 = p1[1];
      wp[v][0] = a0.x; wp[v][1] = a0.y; wp[v][2] = a0.z; wp[v][3] = a0.w;
      wp[v][4] = a1.x; wp[v][5] = a1.y; wp[v][6] = a1.z; wp[v][7] = a1.w;
      wn[v][0] = b0.x; wn[v][1] = b0.y; wn[v][2] = b0.z; wn[v][3] = b0.w;
      wn[v][4] = b1.x; wn[v][5] = b1.y; wn[v][6] = b1.z; wn[v][7] = b1.w;
    }
  }
  pdl_wait();
  float yv[kRowVec][8], rv[kRowVec][8];
  float ss = 0.0f;
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
      unpack8(reinterpret_cast<const uint4*>(y + (size_t)row * H)[vi], yv[v]);
      const float4* rp = reinterpret_cast<const float4*>(r + (size_t)row * H + vi * 8);
      const float4 r0 = rp[0], r1 = rp[1];
      rv[v][0] = r0.x; rv[v][1] = r0.y; rv[v][2] = r0.z; rv[v][3] = r0.w;
      rv[v][4] = r1.x; rv[v][5] = r1.y; rv[v][6] = r1.z; rv[v][7] = r1.w;
#pragma unroll
      for (int e = 0; e < 8; ++e) ss += yv[v][e] * yv[v][e];
    }
  }
  const float inv_y = 1.0f / sqrtf(block_sum(ss, red) / (float)H + eps);
  float ss2 = 0.0f;
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
#pragma unroll
      for (int e = 0; e < 8; ++e) {
        rv[v][e] += yv[v][e] * inv_y * wp[v][e];
        ss2 += rv[v][e] * rv[v][e];
      }
      float4* rp = reinterpret_cast<float4*>(r + (size_t)row * H + vi * 8);
      rp[0] = make_float4(rv[v][0], rv[v][1], rv[v][2], rv[v][3]);
      rp[1] = make_float4(rv[v][4], rv[v][5], rv[v][6], rv[v][7]);
    }
  }
  const float inv_r = 1.0f / sqrtf(block_sum(ss2, red) / (float)H + eps);
#pragma unroll
  for (int v = 0; v < kRowVec; ++v) {
    const int vi = threadIdx.x + v * kRowThreads;
    if (vi < nv) {
      float out[8];
#pragma unroll
      for (int e = 0; e < 8; ++e) out[e] = rv[v][e] * inv_r * wn[v][e];
      reinterpret_cast<uint4*>(a + (size_t)row * H)[vi] = pack8(out);
      if (rq.inv_delta) round8_bf16(out, yv[v]);  // yv now holds the bf16 row
    }
  }
  if (rq.inv_delta) row_quantize(rq, row, H, yv, red);
}

// One warp per head of a row (q heads, then k heads, then v heads).  hd == 256: lane l holds
// dims 4l..4l+3 and 128+4l..128+4l+3, i.e. the four RoPE pairs (i, i + 128), i = 4l..4l+3.
__global__ void qk_rope_kernel(const uint16_t* __restrict__ qkv, AttnShape s, const int* __restrict__ pos0,
                               const float* __restrict__ qn, const float* __restrict__ kn, float eps,
                               const float* __restrict__ rope_cos, const float* __restrict__ rope_sin,
                               float* __restrict__ q, uint16_t* __restrict__ kcache, uint16_t* __restrict__ vcache) {
  pdl_trigger();
  pdl_wait();
  const int row = blockIdx.x;
  const int b = row / s.T, t = row - (row / s.T) * s.T;
  const int pos = *pos0 + t;
  const int head = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hd = s.hd, half = hd >> 1;
  const int qkv_dim = (s.n_q + 2 * s.n_kv) * hd;
  const uint16_t* src = qkv + (size_t)row * qkv_dim + (size_t)head * hd;
  float x1[4], x2[4];
  {
    const uint2 a = *reinterpret_cast<const uint2*>(src + 4 * lane);
    const uint2 c = *reinterpret_cast<const uint2*>(src + half + 4 * lane);
    x1[0] = bf16_lo(a.x); x1[1] = bf16_hi(a.x); x1[2] = bf16_lo(a.y); x1[3] = bf16_hi(a.y);
    x2[0] = bf16_lo(c.x); x2[1] = bf16_hi(c.x); x2[2] = bf16_lo(c.y); x2[3] = bf16_hi(c.y);
  }
  const bool is_q = head < s.n_q, is_k = !is_q && head < s.n_q + s.n_kv;
  const size_t cache_row = ((size_t)b * s.max_seq + pos) * (size_t)(s.n_kv * hd);
  if (!is_q && !is_k) {  // v: straight into the cache
    const int vh = head - s.n_q - s.n_kv;
    uint16_t* dst = vcache + cache_row + (size_t)vh * hd;
    *reinterpret_cast<uint2*>(dst + 4 * lane) = *reinterpret_cast<const uint2*>(src + 4 * lane);
    *reinterpret_cast<uint2*>(dst + half + 4 * lane) = *reinterpret_cast<const uint2*>(src + half + 4 * lane);
    return;
  }
  const float* nw = is_q ? qn : kn;
  if (nw) {
    float ss = 0.0f;
#pragma unroll
    for (int e = 0; e < 4; ++e) ss += x1[e] * x1[e] + x2[e] * x2[e];
    const float inv = 1.0f / sqrtf(warp_sum(ss) / (float)hd + eps);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      x1[e] = x1[e] * inv * nw[4 * lane + e];
      x2[e] = x2[e] * inv * nw[half + 4 * lane + e];
    }
  }
  float y1[4], y2[4];
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float c = rope_cos[(size_t)pos * half + 4 * lane + e], sn = rope_sin[(size_t)pos * half + 4 * lane + e];
    y1[e] = x1[e] * c - x2[e] * sn;
    y2[e] = x2[e] * c + x1[e] * sn;
  }
  if (is_q) {
    float* dst = q + (size_t)row * (s.n_q * hd) + (size_t)head * hd;
    *reinterpret_cast<float4*>(dst + 4 * lane) = make_float4(y1[0], y1[1], y1[2], y1[3]);
    *reinterpret_cast<float4*>(dst + half + 4 * lane) = make_float4(y2[0], y2[1], y2[2], y2[3]);
  } else {
    const int kh = head - s.n_q;
    uint16_t* dst = kcache + cache_row + (size_t)kh * hd;
    uint2 u1, u2;
    u1.x = (uint32_t)f32_to_bf16_bits(y1[0]) | ((uint32_t)f32_to_bf16_bits(y1[1]) << 16);
    u1.y = (uint32_t)f32_to_bf16_bits(y1[2]) | ((uint32_t)f32_to_bf16_bits(y1[3]) << 16);
    u2.x = (uint32_t)f32_to_bf16_bits(y2[0]) | ((uint32_t)f32_to_bf16_bits(y2[1]) << 16);
    u2.y = (uint32_t)f32_to_bf16_bits(y2[2]) | ((uint32_t)f32_to_bf16_bits(y2[3]) << 16);
    *reinterpret_cast<uint2*>(dst + 4 * lane) = u1;
    *reinterpret_cast<uint2*>(dst + half + 4 * lane) = u2;
  }
}

// ---------------------------------------------------------------------------------- attention
constexpr int kKeyTile = 32;
constexpr int kHd = 256;
constexpr int kKStride = kHd + 8;                           // key rows padded to 528 bytes (see below)
constexpr int kKTileBytes = kKeyTile * kKStride * 2;        // one key tile, bf16
constexpr int kVTileBytes = kKeyTile * kHd * 2;             // one value tile, bf16
constexpr int kBufBytes = kKTileBytes + kVTileBytes;
constexpr int kMaxGroup = 8;                                // query heads per key/value head
constexpr int kAttnSmem = 2 * kBufBytes + kMaxGroup * kHd * 4;  // two buffers + the scaled queries
constexpr int kPartStride = kHd + 4;  // floats per split partial: o[256], m, l, 2 pad (16-byte multiple)
constexpr int kMinSplitKeys = 64;     // a key-range split covers at least this many keys

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}

// grid (splits, rows, n_kv), block 32 * G (G = n_q / n_kv query heads sharing one key/value head).
// Warp h handles query head kvh * G + h.  Key/value tiles of 32 positions are copied into shared
// memory asynchronously, two buffers deep (the next tile's copies are in flight while the current
// one is used).  Scores: lane j computes the whole dot product of the query with key j of the
// tile (the query, scaled, is read from shared memory as a broadcast; key rows are padded to 528
// bytes so that the 8 lanes of a shared-memory phase read 8 different 16-byte bank groups).
// Output: lane l accumulates dims 8l .. 8l+7 over the tile's keys.
__global__ void __launch_bounds__(256) attention_kernel(const float* __restrict__ q, const uint16_t* __restrict__ kcache,
                                                        const uint16_t* __restrict__ vcache, AttnShape s,
                                                        const int* __restrict__ pos0, uint16_t* __restrict__ o,
                                                        float* __restrict__ part, unsigned int* __restrict__ ctr) {
  extern __shared__ __align__(16) uint8_t att_smem[];
  __shared__ int s_last;
  pdl_trigger();
  pdl_wait();
  const int split = blockIdx.x, row = blockIdx.y, kvh = blockIdx.z;
  const int G = blockDim.x >> 5;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int head = kvh * G + warp;
  const int b = row / s.T, t = row - (row / s.T) * s.T;
  const int pos = *pos0 + t;
  const int lo = s.window > 0 ? max(0, pos - s.window + 1) : 0;
  const int len = pos - lo + 1;
  // Splits actually used by this row: at least kMinSplitKeys keys each, at most the grid's; the
  // rest of the grid's CTAs for this row have nothing to do.
  const int S = max(1, min((int)gridDim.x, (len + kMinSplitKeys - 1) / kMinSplitKeys));
  if (split >= S) return;
  const int chunk = (len + S - 1) / S;
  const int kb = lo + split * chunk, ke = min(pos + 1, kb + chunk);
  const size_t seq_base = ((size_t)b * s.max_seq) * (size_t)(s.n_kv * kHd) + (size_t)kvh * kHd;
  const uint32_t sbase = smem_u32(att_smem);
  auto stage = [&](int buf, int j0) {
    const int nk = min(kKeyTile, ke - j0);
    const uint32_t kd = sbase + (uint32_t)(buf * kBufBytes), vd = kd + kKTileBytes;
    for (int i = threadIdx.x; i < nk * (kHd / 8); i += blockDim.x) {
      const int jj = i / (kHd / 8), c = i - jj * (kHd / 8);
      const size_t off = seq_base + (size_t)(j0 + jj) * (s.n_kv * kHd) + 8 * c;
      cp_async16(kd + (uint32_t)((jj * kKStride + 8 * c) * 2), kcache + off);
      cp_async16(vd + (uint32_t)((jj * kHd + 8 * c) * 2), vcache + off);
    }
    cp_async_commit();
  };
  if (kb < ke) stage(0, kb);

  // this warp's query, scaled, in shared memory (read back as a broadcast)
  float* qs = reinterpret_cast<float*>(att_smem + 2 * kBufBytes) + warp * kHd;
  {
    const float4* qp = reinterpret_cast<const float4*>(q + (size_t)row * (s.n_q * kHd) + (size_t)head * kHd + 8 * lane);
    const float4 a = qp[0], c = qp[1];
    reinterpret_cast<float4*>(qs + 8 * lane)[0] = make_float4(a.x * s.scale, a.y * s.scale, a.z * s.scale, a.w * s.scale);
    reinterpret_cast<float4*>(qs + 8 * lane)[1] = make_float4(c.x * s.scale, c.y * s.scale, c.z * s.scale, c.w * s.scale);
  }
  __syncwarp();
  float m = -INFINITY, l = 0.0f, acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  int tile = 0;
  for (int j0 = kb; j0 < ke; j0 += kKeyTile, ++tile) {
    const int nk = min(kKeyTile, ke - j0);
    if (j0 + kKeyTile < ke) {
      stage((tile + 1) & 1, j0 + kKeyTile);
      cp_async_wait<1>();
    } else {
      cp_async_wait<0>();
    }
    __syncthreads();
    const uint8_t* buf = att_smem + (tile & 1) * kBufBytes;
    const uint16_t* ks = reinterpret_cast<const uint16_t*>(buf);
    const uint16_t* vs = reinterpret_cast<const uint16_t*>(buf + kKTileBytes);
    float sc = -INFINITY;  // lane j: the score of key j
    if (lane < nk) {
      const uint4* kr = reinterpret_cast<const uint4*>(ks + lane * kKStride);
      float d[4] = {0.0f, 0.0f, 0.0f, 0.0f};  // four partial sums, added in a fixed order
#pragma unroll 8
      for (int c = 0; c < kHd / 8; ++c) {
        float kx[8];
        unpack8(kr[c], kx);
        const float4 q0 = reinterpret_cast<const float4*>(qs + 8 * c)[0];
        const float4 q1 = reinterpret_cast<const float4*>(qs + 8 * c)[1];
        float& dd = d[c & 3];
        dd = fmaf(q0.x, kx[0], dd);
        dd = fmaf(q0.y, kx[1], dd);
        dd = fmaf(q0.z, kx[2], dd);
        dd = fmaf(q0.w, kx[3], dd);
        dd = fmaf(q1.x, kx[4], dd);
        dd = fmaf(q1.y, kx[5], dd);
        dd = fmaf(q1.z, kx[6], dd);
        dd = fmaf(q1.w, kx[7], dd);
      }
      sc = (d[0] + d[1]) + (d[2] + d[3]);
    }
    float tmax = sc;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) tmax = fmaxf(tmax, __shfl_xor_sync(0xffffffffu, tmax, off));
    const float m_new = fmaxf(m, tmax);
    const float corr = expf(m - m_new);  // 0 on the first tile (m = -inf)
    const float p = lane < nk ? expf(sc - m_new) : 0.0f;
    l = l * corr + warp_sum(p);
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] *= corr;
#pragma unroll 4
    for (int jj = 0; jj < nk; ++jj) {
      const float pj = __shfl_sync(0xffffffffu, p, jj);
      float vx[8];
      unpack8(reinterpret_cast<const uint4*>(vs + jj * kHd)[lane], vx);
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = fmaf(pj, vx[e], acc[e]);
    }
    m = m_new;
    __syncthreads();  // this buffer is refilled two tiles later
  }

  uint16_t* out = o + (size_t)row * (s.n_q * kHd) + (size_t)head * kHd + 8 * lane;
  if (S == 1) {
    float y[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) y[e] = acc[e] / l;
    *reinterpret_cast<uint4*>(out) = pack8(y);
    return;
  }
  // partial (m, l, acc) of this split; the last CTA of (row, kvh) combines
  float* pp = part + (((size_t)row * s.n_q + head) * gridDim.x + split) * kPartStride;
  reinterpret_cast<float4*>(pp + 8 * lane)[0] = make_float4(acc[0], acc[1], acc[2], acc[3]);
  reinterpret_cast<float4*>(pp + 8 * lane)[1] = make_float4(acc[4], acc[5], acc[6], acc[7]);
  if (lane == 0) {
    pp[kHd] = m;
    pp[kHd + 1] = l;
  }
  __threadfence();
  __syncthreads();
  if (threadIdx.x == 0) {
    unsigned int* c = ctr + (size_t)row * s.n_kv + kvh;
    const unsigned int prev = atomicAdd(c, 1u);
    s_last = prev == (unsigned int)(S - 1);
    if (s_last) *c = 0u;
  }
  __syncthreads();
  if (!s_last) return;
  __threadfence();
  // Combine: lane sp reads split sp's (m, l); every lane then reads its 8 outputs of all splits,
  // four splits' loads in flight at a time.
  const float* base = part + ((size_t)row * s.n_q + head) * gridDim.x * kPartStride;
  const float ms = lane < S ? __ldcg(base + (size_t)lane * kPartStride + kHd) : -INFINITY;
  const float ls = lane < S ? __ldcg(base + (size_t)lane * kPartStride + kHd + 1) : 0.0f;
  float mx = ms;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, off));
  const float fs = ms == -INFINITY ? 0.0f : expf(ms - mx);  // an empty split weighs nothing
  const float L = warp_sum(ls * fs);
  float y[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int s0 = 0; s0 < S; s0 += 4) {
    float4 va[4], vb[4];
    float f[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int sp = min(s0 + j, S - 1);
      const float4* ps = reinterpret_cast<const float4*>(base + (size_t)sp * kPartStride + 8 * lane);
      va[j] = __ldcg(ps);
      vb[j] = __ldcg(ps + 1);
      f[j] = __shfl_sync(0xffffffffu, fs, sp);
      if (s0 + j >= S) f[j] = 0.0f;
    }
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      y[0] += va[j].x * f[j]; y[1] += va[j].y * f[j]; y[2] += va[j].z * f[j]; y[3] += va[j].w * f[j];
      y[4] += vb[j].x * f[j]; y[5] += vb[j].y * f[j]; y[6] += vb[j].z * f[j]; y[7] += vb[j].w * f[j];
    }
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) y[e] /= L;
  *reinterpret_cast<uint4*>(out) = pack8(y);
}

__global__ void rope_table_kernel(float* cos_t, float* sin_t, int max_seq, int half, int hd, double base) {
  const int idx = blockIdx.x * blockDim.x + threadIdx.x;
  if (idx >= max_seq * half) return;
  const int pos = idx / half, i = idx - (idx / half) * half;
  const double inv_freq = pow(base, -2.0 * (double)i / (double)hd);
  const double ang = (double)pos * inv_freq;
  cos_t[idx] = (float)cos(ang);
  sin_t[idx] = (float)sin(ang);
}

__global__ void set_int_kernel(int* dst, int v) { *dst = v; }

int attention_splits(const AttnShape& s, int sm_count) {
  const int rows = s.B * s.T * s.n_kv;
  if (rows >= 2 * sm_count) return 1;
  const int want = (2 * sm_count + rows - 1) / rows;
  return std::max(1, std::min(32, want));
}

}  // namespace

w8a8_status launch_embed_norm(const int32_t* tokens, int M, const uint16_t* embed, int vocab, int H, float embed_scale,
                              const float* w, float eps, float* r, uint16_t* a, cudaStream_t st, const float* q_inv_delta,
                              uint16_t* q_codes, float* q_sx, int* q_sum) {
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(H % 8 == 0 && H <= 8 * kRowVec * kRowThreads, W8A8_ERR_SHAPE, "embed: hidden %d unsupported", H);
  W8A8_CUDA(launch_pdl(embed_norm_kernel, dim3(M), dim3(kRowThreads), 0, st, tokens, vocab, embed, H, embed_scale, w,
                       eps, r, a, RowQuant{q_inv_delta, q_codes, q_sx, q_sum}));
  return W8A8_OK;
}

w8a8_status launch_residual_norm(const uint16_t* y, int M, int H, const float* w_post, const float* w_next, float eps,
                                 float* r, uint16_t* a, cudaStream_t st, const float* q_inv_delta, uint16_t* q_codes,
                                 float* q_sx, int* q_sum) {
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(H % 8 == 0 && H <= 8 * kRowVec * kRowThreads, W8A8_ERR_SHAPE, "residual norm: hidden %d unsupported", H);
  W8A8_CUDA(launch_pdl(residual_norm_kernel, dim3(M), dim3(kRowThreads), 0, st, y, H, w_post, w_next, eps, r, a,
                       RowQuant{q_inv_delta, q_codes, q_sx, q_sum}));
  return W8A8_OK;
}

w8a8_status launch_qk_rope(const uint16_t* qkv, const AttnShape& s, const int* pos0, const float* qn, const float* kn,
                           float eps, const float* rope_cos, const float* rope_sin, float* q, uint16_t* kcache,
                           uint16_t* vcache, cudaStream_t st) {
  const int M = s.B * s.T;
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(s.hd == kHd && s.n_q + 2 * s.n_kv <= 32, W8A8_ERR_SHAPE, "qk_rope: head_dim %d / heads unsupported", s.hd);
  W8A8_CUDA(launch_pdl(qk_rope_kernel, dim3(M), dim3(32 * (s.n_q + 2 * s.n_kv)), 0, st, qkv, s, pos0, qn, kn, eps,
                       rope_cos, rope_sin, q, kcache, vcache));
  return W8A8_OK;
}

// Workspace: [kAttnCounterBytes of per-(row, kv head) arrival counters, zero between calls | partials]
constexpr size_t kAttnCounterBytes = 65536;

size_t attention_workspace_bytes(const AttnShape& s, int sm_count) {
  const size_t rows = (size_t)s.B * s.T;
  const int S = attention_splits(s, sm_count);
  const size_t partial = S > 1 ? rows * s.n_q * S * kPartStride * 4 : 0;
  return kAttnCounterBytes + partial;
}

w8a8_status launch_attention(const float* q, const uint16_t* kcache, const uint16_t* vcache, const AttnShape& s,
                             const int* pos0, int max_pos_hint, uint16_t* o, void* ws, int sm_count, cudaStream_t st) {
  (void)max_pos_hint;
  const int M = s.B * s.T;
  if (M == 0) return W8A8_OK;
  W8A8_CHECK_ARG(s.hd == kHd && s.n_kv > 0 && s.n_q % s.n_kv == 0 && s.n_q / s.n_kv <= kMaxGroup, W8A8_ERR_SHAPE,
                 "attention: head layout unsupported");
  W8A8_CHECK_ARG((size_t)M * s.n_kv * 4 <= kAttnCounterBytes, W8A8_ERR_SHAPE, "attention: %d rows exceed the counters",
                 M);
  const int S = attention_splits(s, sm_count);
  unsigned int* ctr = reinterpret_cast<unsigned int*>(ws);
  float* part = reinterpret_cast<float*>(reinterpret_cast<char*>(ws) + kAttnCounterBytes);
  dim3 grid(S, M, s.n_kv);
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(attention_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kAttnSmem));
    attr_set[dev] = true;
  }
  W8A8_CUDA(launch_pdl(attention_kernel, grid, dim3(32 * (s.n_q / s.n_kv)), (size_t)kAttnSmem, st, q, kcache, vcache, s,
                       pos0, o, part, ctr));
  return W8A8_OK;
}

w8a8_status launch_rope_table(float* cos_t, float* sin_t, int max_seq, int hd, double base, cudaStream_t st) {
  const int half = hd / 2;
  const int n = max_seq * half;
  rope_table_kernel<<<(n + 255) / 256, 256, 0, st>>>(cos_t, sin_t, max_seq, half, hd, base);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

w8a8_status launch_set_int(int* dst, int value, cudaStream_t st) {
  set_int_kernel<<<1, 1, 0, st>>>(dst, value);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

}  // namespace w8a8
