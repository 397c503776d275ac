// Prefill attention (many new tokens per sequence) on the tensor cores, flash-attention style.
//
// The query-row kernel (attention_kernel) reads a row's keys and values from L2 for every query
// row, so a 2048-token prefill moves about 2 GB per layer through L2 and the arithmetic runs on
// the CUDA cores.  Here a CTA takes a block of 64 queries of one head and walks the keys in tiles
// of 32 positions that all of its queries share:
//  * grid (query blocks, query heads, sequences), 8 warps in two groups of four; warp w of a group
//    owns query rows 16w .. 16w+15 of the block, group 0 takes the even key tiles and group 1 the
//    odd ones (two warps per SM sub-partition, each with half of the serial MMA chain), and at the
//    end group 0 merges group 1's (m, l, O) through shared memory.  The block's queries (after QK-norm and RoPE, fp32) are scaled by the
//    attention scale and rounded to fp16 into shared memory once (fp16, not bf16: 11 mantissa
//    bits keep the scores and probabilities close to the fp32 arithmetic of the other paths);
//  * key/value tiles (bf16 rows of 512 bytes straight from the cache) arrive by cp.async, two
//    tiles deep per group, into shared memory whose 16-byte chunks are XOR-swizzled by (row mod 8), so the
//    8 row addresses of an ldmatrix phase hit 8 different bank groups; each landed tile is
//    converted to fp16 in place (exact for the cache's bf16 values in the fp16 normal range);
//  * S = Q K^T with mma.sync m16n8k16 (fp16 in, fp32 accumulation): Q fragments by ldmatrix, K
//    fragments by ldmatrix on key rows (K rows are the column-major B operand as stored);
//  * causal and sliding-window masks per element (key j is visible to the query at position p
//    when lo(p) <= j <= p), then the online softmax per row (running max m and sum l, fp32), P
//    rounded to fp16 in registers (the accumulator layout of S is the A-operand layout of the
//    next MMA), O += P V with V fragments by ldmatrix.trans;
//  * finally o = O / l rounded to bf16.
#include <cmath>

#include "decoder_kernels.cuh"

namespace w8a8 {

namespace {

constexpr int kHd = 256;
constexpr int kBq = 64;             // queries per CTA
constexpr int kBk = 32;             // keys per tile
constexpr int kGW = kBq / 16;       // warps per group (one per 16 query rows)
constexpr int kWarps = 2 * kGW;     // two groups: even and odd key tiles
constexpr int kGT = kGW * 32;       // threads per group
constexpr int kRowBytes = kHd * 2;  // one bf16 row of 256
constexpr int kTileBytes = kBk * kRowBytes;
constexpr int kOffQ = 0;
constexpr int kOffKV = kBq * kRowBytes;                 // per group two buffers of (K tile, V tile)
constexpr int kGroupKV = 2 * 2 * kTileBytes;
constexpr int kSmem = kOffKV + 2 * kGroupKV;            // 32 KB + 128 KB
static_assert(kGW * 32 * 132 * 4 <= 2 * kGroupKV, "the merge area must fit in the key/value buffers");

__device__ __forceinline__ uint32_t swz(int row, int chunk) {  // byte offset of a 16-byte chunk
  return (uint32_t)(row * kRowBytes + ((chunk ^ (row & 7)) << 4));
}
__device__ __forceinline__ void ldsm_x4(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.shared.b16 {%0, %1, %2, %3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void ldsm_x4_t(uint32_t addr, uint32_t& r0, uint32_t& r1, uint32_t& r2, uint32_t& r3) {
  asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0, %1, %2, %3}, [%4];\n"
               : "=r"(r0), "=r"(r1), "=r"(r2), "=r"(r3)
               : "r"(addr));
}
__device__ __forceinline__ void cp16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp16_zero(uint32_t dst) {  // a 16-byte chunk of zeros (rows past the range)
  asm volatile("st.shared.v4.u32 [%0], {%1, %1, %1, %1};\n" ::"r"(dst), "r"(0u) : "memory");
}
__device__ __forceinline__ uint32_t pack_bf16(float a, float b) {
  return (uint32_t)f32_to_bf16_bits(a) | ((uint32_t)f32_to_bf16_bits(b) << 16);
}
__device__ __forceinline__ uint32_t pack_f16(float a, float b) {  // a in the low half
  uint32_t r;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;\n" : "=r"(r) : "f"(b), "f"(a));
  return r;
}
__device__ __forceinline__ uint32_t bf16x2_to_f16x2(uint32_t w) {
  return pack_f16(__uint_as_float(w << 16), __uint_as_float(w & 0xFFFF0000u));
}

__global__ void __launch_bounds__(kWarps * 32) attn_prefill_kernel(const float* __restrict__ q,
                                                                   const uint16_t* __restrict__ kcache,
                                                                   const uint16_t* __restrict__ vcache, AttnShape s,
                                                                   const int* __restrict__ pos0,
                                                                   uint16_t* __restrict__ o) {
  extern __shared__ __align__(128) uint8_t smem[];
  pdl_trigger();
  pdl_wait();
  const int qb = blockIdx.x, head = blockIdx.y, b = blockIdx.z;
  const int G = s.n_q / s.n_kv, kvh = head / G;
  const int warp_all = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int grp = warp_all / kGW, warp = warp_all % kGW, gt = threadIdx.x % kGT;
  const int g = lane >> 2, t4 = lane & 3;
  const int p0 = *pos0;
  const int t0 = qb * kBq;                           // first query (token index within the call)
  const int t_last = min(s.T, t0 + kBq) - 1;
  const int hi = p0 + t_last;                        // last key any query of the block sees
  const int lo = s.window > 0 ? max(0, p0 + t0 - s.window + 1) : 0;  // first key any query sees
  const uint32_t sb = smem_u32(smem);
  const size_t row_stride = (size_t)s.n_kv * kHd;
  const size_t seq_base = (size_t)b * s.max_seq * row_stride + (size_t)kvh * kHd;

  // key/value tile starting at key j0 into this group's buffer buf (keys past hi: zeros)
  auto stage = [&](int buf, int j0) {
    const uint32_t kd = sb + kOffKV + (uint32_t)(grp * kGroupKV + buf * 2 * kTileBytes), vd = kd + kTileBytes;
    for (int i = gt; i < kBk * (kHd / 8); i += kGT) {
      const int r = i >> 5, c = i & 31, j = j0 + r;
      if (j <= hi) {
        const size_t off = seq_base + (size_t)j * row_stride + 8 * c;
        cp16(kd + swz(r, c), kcache + off);
        cp16(vd + swz(r, c), vcache + off);
      } else {
        cp16_zero(kd + swz(r, c));
        cp16_zero(vd + swz(r, c));
      }
    }
    asm volatile("cp.async.commit_group;\n" ::: "memory");
  };
  const int jt0 = lo & ~(kBk - 1);  // tiles aligned to 32 keys; group grp takes tiles grp, grp + 2, ...
  if (jt0 + grp * kBk <= hi) stage(0, jt0 + grp * kBk);

  // the block's queries, scaled, as fp16 (rows past the call's tokens: zeros)
  for (int i = threadIdx.x; i < kBq * (kHd / 8); i += kWarps * 32) {
    const int r = i >> 5, c = i & 31, t = t0 + r;
    uint4 w = make_uint4(0u, 0u, 0u, 0u);
    if (t < s.T) {
      const float4* src = reinterpret_cast<const float4*>(q + ((size_t)b * s.T + t) * (s.n_q * kHd) +
                                                          (size_t)head * kHd + 8 * c);
      const float4 a = src[0], d = src[1];
      w.x = pack_f16(a.x * s.scale, a.y * s.scale);
      w.y = pack_f16(a.z * s.scale, a.w * s.scale);
      w.z = pack_f16(d.x * s.scale, d.y * s.scale);
      w.w = pack_f16(d.z * s.scale, d.w * s.scale);
    }
    *reinterpret_cast<uint4*>(smem + kOffQ + swz(r, c)) = w;
  }

  // this thread's two query rows (g and g + 8 of the warp's 16) and their visible key ranges
  const int ra = 16 * warp + g, rb = ra + 8;
  const int pa = p0 + t0 + ra, pb = p0 + t0 + rb;
  const int loa = s.window > 0 ? max(0, pa - s.window + 1) : 0;
  const int lob = s.window > 0 ? max(0, pb - s.window + 1) : 0;
  float O[kHd / 8][4];
#pragma unroll
  for (int n = 0; n < kHd / 8; ++n) O[n][0] = O[n][1] = O[n][2] = O[n][3] = 0.0f;
  float ma = -INFINITY, mb = -INFINITY, la = 0.0f, lb = 0.0f;
  const uint32_t qbase = sb + kOffQ;
  __syncthreads();  // the queries are in shared memory
  auto group_sync = [&]() { named_bar_sync(1 + grp, kGT); };

  int buf = 0;
  for (int j0 = jt0 + grp * kBk; j0 <= hi; j0 += 2 * kBk, buf ^= 1) {
    if (j0 + 2 * kBk <= hi) {
      stage(buf ^ 1, j0 + 2 * kBk);
      asm volatile("cp.async.wait_group 1;\n" ::: "memory");
    } else {
      asm volatile("cp.async.wait_group 0;\n" ::: "memory");
    }
    group_sync();
    const uint32_t kbase = sb + kOffKV + (uint32_t)(grp * kGroupKV + buf * 2 * kTileBytes), vbase = kbase + kTileBytes;
    {  // the landed K and V tiles, bf16 -> fp16 in place
      uint8_t* kv = smem + kOffKV + grp * kGroupKV + buf * 2 * kTileBytes;
      for (int i = gt; i < 2 * kTileBytes / 16; i += kGT) {
        uint4* pchunk = reinterpret_cast<uint4*>(kv + 16 * i);
        uint4 w = *pchunk;
        w.x = bf16x2_to_f16x2(w.x);
        w.y = bf16x2_to_f16x2(w.y);
        w.z = bf16x2_to_f16x2(w.z);
        w.w = bf16x2_to_f16x2(w.w);
        *pchunk = w;
      }
      group_sync();
    }

    // S = Q K^T for the warp's 16 rows x 32 keys (4 n-tiles of 8 keys)
    float S[kBk / 8][4];
#pragma unroll
    for (int n = 0; n < kBk / 8; ++n) S[n][0] = S[n][1] = S[n][2] = S[n][3] = 0.0f;
#pragma unroll 4
    for (int kk = 0; kk < kHd / 16; ++kk) {
      uint32_t a0, a1, a2, a3;
      ldsm_x4(qbase + swz(16 * warp + (lane & 15), 2 * kk + (lane >> 4)), a0, a1, a2, a3);
#pragma unroll
      for (int p = 0; p < kBk / 16; ++p) {  // n-tiles 2p and 2p + 1
        const int key = 16 * p + (lane & 7) + ((lane >> 4) << 3);
        const int chunk = 2 * kk + ((lane >> 3) & 1);
        uint32_t b0, b1, b2, b3;
        ldsm_x4(kbase + swz(key, chunk), b0, b1, b2, b3);
        mma_f16_16816(S[2 * p], a0, a1, a2, a3, b0, b1);
        mma_f16_16816(S[2 * p + 1], a0, a1, a2, a3, b2, b3);
      }
    }

    // masks and the online softmax (rows ra: S[n][0..1], rb: S[n][2..3])
    float ta = -INFINITY, tb = -INFINITY;
#pragma unroll
    for (int n = 0; n < kBk / 8; ++n) {
#pragma unroll
      for (int e = 0; e < 2; ++e) {
        const int j = j0 + 8 * n + 2 * t4 + e;
        if (j < loa || j > pa) S[n][e] = -INFINITY;
        if (j < lob || j > pb) S[n][2 + e] = -INFINITY;
        ta = fmaxf(ta, S[n][e]);
        tb = fmaxf(tb, S[n][2 + e]);
      }
    }
    ta = fmaxf(ta, __shfl_xor_sync(0xffffffffu, ta, 1));
    ta = fmaxf(ta, __shfl_xor_sync(0xffffffffu, ta, 2));
    tb = fmaxf(tb, __shfl_xor_sync(0xffffffffu, tb, 1));
    tb = fmaxf(tb, __shfl_xor_sync(0xffffffffu, tb, 2));
    const float na = fmaxf(ma, ta), nb = fmaxf(mb, tb);
    // rows with no visible key yet keep m = -inf: scale 1, probabilities 0
    const float ca = na == -INFINITY ? 1.0f : expf(ma - na), cb = nb == -INFINITY ? 1.0f : expf(mb - nb);
    float sa = 0.0f, sbm = 0.0f;
    uint32_t P[kBk / 8][2];  // fp16 pairs: P[n][0] row ra, P[n][1] row rb
#pragma unroll
    for (int n = 0; n < kBk / 8; ++n) {
      const float e0 = na == -INFINITY ? 0.0f : expf(S[n][0] - na);
      const float e1 = na == -INFINITY ? 0.0f : expf(S[n][1] - na);
      const float e2 = nb == -INFINITY ? 0.0f : expf(S[n][2] - nb);
      const float e3 = nb == -INFINITY ? 0.0f : expf(S[n][3] - nb);
      sa += e0 + e1;
      sbm += e2 + e3;
      P[n][0] = pack_f16(e0, e1);
      P[n][1] = pack_f16(e2, e3);
    }
    sa += __shfl_xor_sync(0xffffffffu, sa, 1);
    sa += __shfl_xor_sync(0xffffffffu, sa, 2);
    sbm += __shfl_xor_sync(0xffffffffu, sbm, 1);
    sbm += __shfl_xor_sync(0xffffffffu, sbm, 2);
    la = la * ca + sa;
    lb = lb * cb + sbm;
    ma = na;
    mb = nb;
#pragma unroll
    for (int n = 0; n < kHd / 8; ++n) {
      O[n][0] *= ca;
      O[n][1] *= ca;
      O[n][2] *= cb;
      O[n][3] *= cb;
    }

    // O += P V: k-steps of 16 keys, 32 n-tiles of 8 dims
#pragma unroll
    for (int kk = 0; kk < kBk / 16; ++kk) {
      const uint32_t a0 = P[2 * kk][0], a1 = P[2 * kk][1], a2 = P[2 * kk + 1][0], a3 = P[2 * kk + 1][1];
      const int key = 16 * kk + (lane & 7) + (((lane >> 3) & 1) << 3);
#pragma unroll
      for (int d = 0; d < kHd / 16; ++d) {  // dims 16d .. 16d + 15: n-tiles 2d and 2d + 1
        uint32_t b0, b1, b2, b3;
        ldsm_x4_t(vbase + swz(key, 2 * d + (lane >> 4)), b0, b1, b2, b3);
        mma_f16_16816(O[2 * d], a0, a1, a2, a3, b0, b1);
        mma_f16_16816(O[2 * d + 1], a0, a1, a2, a3, b2, b3);
      }
    }
    group_sync();  // the buffer is refilled two of this group's tiles on
  }

  // group 1 hands its (m, l, O) to group 0 through the key/value area (now free), laid out
  // [value][warp][lane] so that a warp's accesses are consecutive words
  __syncthreads();
  float* xo = reinterpret_cast<float*>(smem + kOffKV);
  const int slot = warp * 32 + lane;
  if (grp == 1) {
#pragma unroll
    for (int n = 0; n < kHd / 8; ++n)
#pragma unroll
      for (int e = 0; e < 4; ++e) xo[(4 * n + e) * kGT + slot] = O[n][e];
    xo[128 * kGT + slot] = ma;
    xo[129 * kGT + slot] = mb;
    xo[130 * kGT + slot] = la;
    xo[131 * kGT + slot] = lb;
  }
  __syncthreads();
  if (grp == 1) return;
  {
    const float ma1 = xo[128 * kGT + slot], mb1 = xo[129 * kGT + slot];
    const float la1 = xo[130 * kGT + slot], lb1 = xo[131 * kGT + slot];
    const float na = fmaxf(ma, ma1), nb = fmaxf(mb, mb1);
    const float fa0 = ma == -INFINITY ? 0.0f : expf(ma - na), fa1 = ma1 == -INFINITY ? 0.0f : expf(ma1 - na);
    const float fb0 = mb == -INFINITY ? 0.0f : expf(mb - nb), fb1 = mb1 == -INFINITY ? 0.0f : expf(mb1 - nb);
    la = la * fa0 + la1 * fa1;
    lb = lb * fb0 + lb1 * fb1;
#pragma unroll
    for (int n = 0; n < kHd / 8; ++n) {
      O[n][0] = O[n][0] * fa0 + xo[(4 * n + 0) * kGT + slot] * fa1;
      O[n][1] = O[n][1] * fa0 + xo[(4 * n + 1) * kGT + slot] * fa1;
      O[n][2] = O[n][2] * fb0 + xo[(4 * n + 2) * kGT + slot] * fb1;
      O[n][3] = O[n][3] * fb0 + xo[(4 * n + 3) * kGT + slot] * fb1;
    }
  }

  // o = O / l (rows past the call's tokens are not stored)
  const int ta_tok = t0 + ra, tb_tok = t0 + rb;
  const float ia = la > 0.0f ? 1.0f / la : 0.0f, ib = lb > 0.0f ? 1.0f / lb : 0.0f;
  uint16_t* oa = o + ((size_t)b * s.T + ta_tok) * (s.n_q * kHd) + (size_t)head * kHd;
  uint16_t* ob = o + ((size_t)b * s.T + tb_tok) * (s.n_q * kHd) + (size_t)head * kHd;
#pragma unroll
  for (int n = 0; n < kHd / 8; ++n) {
    const int col = 8 * n + 2 * t4;
    if (ta_tok < s.T) *reinterpret_cast<uint32_t*>(oa + col) = pack_bf16(O[n][0] * ia, O[n][1] * ia);
    if (tb_tok < s.T) *reinterpret_cast<uint32_t*>(ob + col) = pack_bf16(O[n][2] * ib, O[n][3] * ib);
  }
}

}  // namespace

bool attention_prefill_supported(const AttnShape& s) {
  return s.hd == kHd && s.n_kv > 0 && s.n_q % s.n_kv == 0 && s.T > 1;
}

w8a8_status launch_attention_prefill(const float* q, const uint16_t* kcache, const uint16_t* vcache, const AttnShape& s,
                                     const int* pos0, uint16_t* o, cudaStream_t st) {
  if (s.B == 0 || s.T == 0) return W8A8_OK;
  W8A8_CHECK_ARG(attention_prefill_supported(s), W8A8_ERR_SHAPE, "prefill attention: head dim 256 and T > 1 only");
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(attn_prefill_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem));
    attr_set[dev] = true;
  }
  const dim3 grid((unsigned)((s.T + kBq - 1) / kBq), (unsigned)s.n_q, (unsigned)s.B);
  W8A8_CUDA(launch_pdl(attn_prefill_kernel, grid, dim3(kWarps * 32), (size_t)kSmem, st, q, kcache, vcache, s, pos0, o));
  return W8A8_OK;
}

}  // namespace w8a8
