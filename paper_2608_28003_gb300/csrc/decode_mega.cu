// Persistent decode kernel: all decoder layers of one decode step (batch 1, one new token) in one
// cooperative launch of one CTA per SM.
//
// At one token a layer's five dependent steps (q/k/v projection, attention, o projection, gate/up
// with GeGLU, down) each move a few MB at most, so as separate kernels most of their time is the
// gap between a kernel's end and its successor's start.  Here the steps are phases of one kernel:
//  * every CTA owns a fixed share of the rows of every linear (whole rows: 8-row groups, 16 for
//    gate/up so that a gate row and its up row stay together).  One producer thread streams the
//    CTA's rows of all linears of all layers, in execution order, through a ring of 18 KB stages
//    (8 rows x 2304 bytes: a whole row of K = 1152 in bf16, or a k chunk of longer rows) with bulk
//    async copies.  The weights do not depend on the activations, so the ring runs ahead of the
//    computation across phase and layer boundaries and HBM stays busy while a phase waits;
//  * the 8 consumer warps run the phases.  Phase p of a layer starts when a global counter shows
//    that all CTAs have finished phase p - 1 (each CTA adds 1 after its writes, with a gpu-scope
//    fence before the add and an acquire load on the waiting side; activations are then read from
//    L2, never L1).  Every CTA first rebuilds the phase's input row in shared memory: the
//    residual step of the decoder (residual add, post-norm of the previous sublayer, pre-norm of
//    the next: CTA 0 also writes the updated residual stream, which ping-pongs between two
//    buffers) where one precedes the linear, then K1 for W8A8 sublayers (smoothing by 1 / delta,
//    per-token absmax, INT8 codes: Eq. stx / xint8 of the per-token quantiser);
//  * warp w computes row w of each 8-row stage over the full k range (fp32 FMAs on bf16, or dp4a
//    with exact INT32 sums, Eq. gemm-final), lanes reading consecutive 16-byte pieces; a butterfly
//    ends the sum and lane 0 writes the output: bf16 (dequantised fl(fl(s_x s_w) acc) for W8A8),
//    or for gate/up the GeGLU of the row pair;
//  * the attention phase runs on n_q x S CTAs (S splits of the key range per query head, S from
//    the context length): QK-norm and RoPE of the query and the new key, the key/value row written
//    to the cache (one CTA per key/value head), scores and an online softmax per warp over its
//    keys, the CTA's partial (m, l, o) to global memory; the last CTA of a head (atomic count)
//    combines the S partials into the head's output.
// Every wait (ring barriers and phase counters) is bounded: on timeout the CTA sets the error word
// and returns, so a failure ends the launch instead of hanging it.
#include "decode_mega.cuh"

namespace w8a8 {

namespace {

constexpr int kCW = 8;                    // consumer warps
constexpr int kThreads = kCW * 32;
constexpr int kHd = 256;
constexpr int kSB = 18432;                // ring stage: 8 rows x 2304 bytes
constexpr int kStages = 9;
constexpr int kMaxK = 7168;
constexpr int kPartF = kHd + 4;           // per-warp attention partial: o[256], m, l, pad
constexpr int kOffX = kStages * kSB;      // the phase's input row, bf16 [kMaxK]
constexpr int kOffXq = kOffX + kMaxK * 2; // its INT8 codes [kMaxK]
constexpr int kOffIdr = kOffXq + kMaxK;   // 1 / delta of the phase's W8A8 linear, fp32 [kMaxK]
constexpr int kOffQ = kOffIdr + kMaxK * 4;  // attention: scaled query fp32 [256]
constexpr int kOffKn = kOffQ + kHd * 4;   // new key bf16 [256]
constexpr int kOffVn = kOffKn + kHd * 2;  // new value bf16 [256]
constexpr int kOffPart = kOffVn + kHd * 2;
constexpr int kSmem = kOffPart + kCW * kPartF * 4;
constexpr int kSmemAlloc = kSmem + 128;   // the ring starts on a 128-byte boundary
constexpr long long kPhaseBudget = kWaitBudgetCycles;

enum Phase { PH_QKV = 0, PH_ATT = 1, PH_O = 2, PH_GU = 3, PH_DOWN = 4 };

__device__ __forceinline__ unsigned int ld_acquire_gpu(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];\n" : "=r"(v) : "l"(p) : "memory");
  return v;
}
// Loads of constants that stay where they are written (a read-only load may be hoisted anywhere,
// which here would keep a whole layer's constants live in registers).
__device__ __forceinline__ float4 ld_f4(const float* p) {
  float4 v;
  asm volatile("ld.global.v4.f32 {%0, %1, %2, %3}, [%4];\n" : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ float ld_f1(const float* p) {
  float v;
  asm volatile("ld.global.f32 %0, [%1];\n" : "=f"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ int warp_sum_i(int v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ void unpack8(const uint4& v, float (&x)[8]) {
  x[0] = bf16_lo(v.x); x[1] = bf16_hi(v.x); x[2] = bf16_lo(v.y); x[3] = bf16_hi(v.y);
  x[4] = bf16_lo(v.z); x[5] = bf16_hi(v.z); x[6] = bf16_lo(v.w); x[7] = bf16_hi(v.w);
}
__device__ __forceinline__ uint4 pack8(const float (&o)[8]) {
  uint4 w;
  w.x = (uint32_t)f32_to_bf16_bits(o[0]) | ((uint32_t)f32_to_bf16_bits(o[1]) << 16);
  w.y = (uint32_t)f32_to_bf16_bits(o[2]) | ((uint32_t)f32_to_bf16_bits(o[3]) << 16);
  w.z = (uint32_t)f32_to_bf16_bits(o[4]) | ((uint32_t)f32_to_bf16_bits(o[5]) << 16);
  w.w = (uint32_t)f32_to_bf16_bits(o[6]) | ((uint32_t)f32_to_bf16_bits(o[7]) << 16);
  return w;
}

// The rows of linear j of layer l that this CTA owns, and how they are staged.
struct Lin {
  const void* w;
  int N, K, kc;     // kc: k elements per stage row
  int g0, g1;       // 8-row groups [g0, g1)
  bool i8;
};
__device__ __forceinline__ Lin lin_of(const MegaArgs& a, const MegaLayer& Ly, int l, int j, int cta, int G) {
  Lin g;
  g.i8 = (((j < 2 ? a.attn_bits : a.ffn_bits) >> l) & 1u) != 0u;
  const int qkv_dim = (a.n_q + 2 * a.n_kv) * kHd;
  g.N = j == 0 ? qkv_dim : j == 1 ? a.H : j == 2 ? 2 * a.F : a.H;
  g.K = j == 0 ? a.H : j == 1 ? a.n_q * kHd : j == 2 ? a.H : a.F;
  const int U = j == 2 ? 16 : 8;  // gate/up: a gate group and its up group together
  const int units = (g.N + U - 1) / U;
  const int u0 = (int)((long long)cta * units / G), u1 = (int)((long long)(cta + 1) * units / G);
  g.g0 = u0 * (U / 8);
  g.g1 = min((g.N + 7) / 8, u1 * (U / 8));
  g.kc = min(g.K, g.i8 ? kSB / 8 : kSB / 16);
  g.w = g.i8 ? (const void*)Ly.w8[j] : (const void*)Ly.w16[j];
  return g;
}

// ------------------------------------------------------------------------------ weight stream
// The CTA's ring stages in execution order: (layer l, linear j, 8-row group grp, k offset k0).
// Every consumer warp walks this sequence twice over: at the stage it consumes, and kStages ahead
// (the stage that will refill the slot it is about to release).
struct Cursor {
  Lin g;
  int l, j, grp, k0;
  bool valid;
};
__device__ __forceinline__ void cursor_settle(const MegaArgs& a, int cta, int G, Cursor& u) {
  // move to the first linear (from (l, j) on) in which this CTA owns rows
  while (u.l < a.L) {
    u.g = lin_of(a, a.layers[u.l], u.l, u.j, cta, G);
    if (u.g.g0 < u.g.g1) {
      u.grp = u.g.g0;
      u.k0 = 0;
      u.valid = true;
      return;
    }
    if (++u.j == 4) {
      u.j = 0;
      ++u.l;
    }
  }
  u.valid = false;
}
__device__ __forceinline__ void cursor_start(const MegaArgs& a, int cta, int G, Cursor& u) {
  u.l = 0;
  u.j = 0;
  cursor_settle(a, cta, G, u);
}
__device__ __forceinline__ void cursor_next(const MegaArgs& a, int cta, int G, Cursor& u) {
  if (!u.valid) return;
  u.k0 += u.g.kc;
  if (u.k0 < u.g.K) return;
  u.k0 = 0;
  if (++u.grp < u.g.g1) return;
  if (++u.j == 4) {
    u.j = 0;
    ++u.l;
  }
  cursor_settle(a, cta, G, u);
}
// Copy stage u into ring slot s (completion counted on full barrier `bar`).
__device__ __forceinline__ void issue_stage(const Cursor& u, uint32_t ring, int s, uint32_t bar) {
  const int esz = u.g.i8 ? 1 : 2;
  const int rows = min(8, u.g.N - 8 * u.grp);
  const uint32_t bytes = (uint32_t)(min(u.g.kc, u.g.K - u.k0) * esz);
  mbar_arrive_expect_tx(bar, (uint32_t)rows * bytes);
  const char* src = reinterpret_cast<const char*>(u.g.w) + ((size_t)8 * u.grp * u.g.K + u.k0) * esz;
  const uint32_t dst = ring + (uint32_t)(s * kSB);
  if (u.g.kc == u.g.K) {  // whole rows: the group is one contiguous block
    bulk_g2s(dst, src, (uint32_t)rows * bytes, bar);
  } else {
    for (int rr = 0; rr < rows; ++rr) bulk_g2s(dst + (uint32_t)rr * bytes, src + (size_t)rr * u.g.K * esz, bytes, bar);
  }
}

// ------------------------------------------------------------------------------ consumers
struct Ctx {
  const MegaArgs* a;
  uint8_t* sm;
  uint32_t ring, full0, empty0, xs, xq;
  int* slot_cnt;     // per ring slot: warps done with it (the last one refills it)
  int* issued;       // stages issued so far, and stages released by all warps (for the drain on
  int* consumed;     // failure: the copies of issued stages must land before the CTA exits)
  Cursor ahead;      // the stage kStages after the one being consumed
  float* red;   // [kCW] reduction slots
  int* flag;    // broadcast of thread 0's wait result
  float* sx;    // the phase's s_x (W8A8)
  int cta, G, tid, warp, lane;
  int s;
  uint32_t ph;
};

// Sum over the 256 consumer threads (lane tree, then warps 0..7 in turn), as the residual-norm
// kernel orders it; every consumer thread gets the result.
__device__ __forceinline__ float consumer_sum(Ctx& c, float v) {
  v = warp_sum_f(v);
  named_bar_sync(1, kCW * 32);
  if (c.lane == 0) c.red[c.warp] = v;
  named_bar_sync(1, kCW * 32);
  float t = 0.0f;
#pragma unroll
  for (int i = 0; i < kCW; ++i) t += c.red[i];
  named_bar_sync(1, kCW * 32);  // the slots are reused
  return t;
}

// Wait until all G CTAs have counted phase `idx` (idx < 0: nothing to wait for).
__device__ __forceinline__ bool wait_phase(Ctx& c, int idx) {
  if (idx < 0) return true;
  if (c.tid == 0) {
    const unsigned int* p = c.a->sync + idx;
    bool ok = ld_acquire_gpu(p) >= (unsigned)c.G;
    if (!ok) {
      const long long t0 = clock64();
      while (!(ok = ld_acquire_gpu(p) >= (unsigned)c.G)) {
        if (clock64() - t0 > kPhaseBudget) break;
        __nanosleep(64);
      }
    }
    if (!ok) atomicOr(c.a->err, DEVERR_CONSUMER_WAIT);
    *c.flag = ok ? 1 : 0;
  }
  named_bar_sync(1, kCW * 32);
  return *c.flag != 0;
}
// True when every consumer thread passes ok (a barrier of the 256 consumer threads).
__device__ __forceinline__ bool consumers_all(bool ok) {
  uint32_t r;
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.u32 p, %1, 0;\n bar.red.and.pred p, 1, %2, p;\n selp.u32 %0, 1, 0, p;\n}\n"
      : "=r"(r)
      : "r"((uint32_t)ok), "r"(kCW * 32)
      : "memory");
  return r != 0;
}
// Count this CTA's phase `idx` as done, unless a warp of the CTA gave up (then the CTA stops).
__device__ __forceinline__ bool count_phase(Ctx& c, int idx, bool ok) {
  if (!consumers_all(ok)) return false;  // also orders every consumer thread's writes before the count
  if (c.tid == 0) {
    __threadfence();
    atomicAdd(c.a->sync + idx, 1u);
  }
  return true;
}

// Residual step into the phase input: r_out = r_in + rmsnorm(y) * w_post; x = bf16(rmsnorm(r_out)
// * w_next) in shared memory; CTA 0 writes r_out.  Thread t < H / 8 owns channels 8t .. 8t+7.
__device__ __forceinline__ void residual_step(Ctx& c, int H, const uint16_t* y, const float* r_in, float* r_out, const float (&wp)[8],
                              const float (&wn)[8]) {
  const float eps = c.a->eps;
  const bool mine = c.tid < (H >> 3);
  float yv[8], rv[8];
  float ss = 0.0f;
  if (mine) {
    unpack8(__ldcg(reinterpret_cast<const uint4*>(y) + c.tid), yv);
    const float4 r0 = __ldcg(reinterpret_cast<const float4*>(r_in + 8 * c.tid));
    const float4 r1 = __ldcg(reinterpret_cast<const float4*>(r_in + 8 * c.tid) + 1);
    rv[0] = r0.x; rv[1] = r0.y; rv[2] = r0.z; rv[3] = r0.w; rv[4] = r1.x; rv[5] = r1.y; rv[6] = r1.z; rv[7] = r1.w;
#pragma unroll
    for (int e = 0; e < 8; ++e) ss += yv[e] * yv[e];
  }
  const float inv_y = 1.0f / sqrtf(consumer_sum(c, ss) / (float)H + eps);
  float ss2 = 0.0f;
  if (mine) {
#pragma unroll
    for (int e = 0; e < 8; ++e) {
      rv[e] += yv[e] * inv_y * wp[e];
      ss2 += rv[e] * rv[e];
    }
    if (c.cta == 0) {
      float4* ro = reinterpret_cast<float4*>(r_out + 8 * c.tid);
      __stcg(ro, make_float4(rv[0], rv[1], rv[2], rv[3]));
      __stcg(ro + 1, make_float4(rv[4], rv[5], rv[6], rv[7]));
    }
  }
  const float inv_r = 1.0f / sqrtf(consumer_sum(c, ss2) / (float)H + eps);
  if (mine) {
    float o[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) o[e] = rv[e] * inv_r * wn[e];
    *reinterpret_cast<uint4*>(c.sm + kOffX + 16 * c.tid) = pack8(o);
  }
  named_bar_sync(1, kCW * 32);
}

// The phase input straight from global memory (bf16 [K]) into shared memory.
__device__ __forceinline__ void input_copy(Ctx& c, const uint16_t* x, int K) {
  const int nv = K >> 3;
  for (int i = c.tid; i < nv; i += 4 * kCW * 32) {  // four loads in flight per thread
    uint4 v[4];
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (i + u * kCW * 32 < nv) v[u] = __ldcg(reinterpret_cast<const uint4*>(x) + i + u * kCW * 32);
#pragma unroll
    for (int u = 0; u < 4; ++u)
      if (i + u * kCW * 32 < nv) *reinterpret_cast<uint4*>(c.sm + kOffX + 16 * (i + u * kCW * 32)) = v[u];
  }
  named_bar_sync(1, kCW * 32);
}

// 1 / delta of the next W8A8 linear into shared memory (cp.async, issued before the phase's wait;
// thread t copies the vectors it reads in quantize_input).
__device__ __forceinline__ void prefetch_idr(Ctx& c, const float* inv_delta, int K) {
  const int nv = K >> 3;
  for (int vi = c.tid; vi < nv; vi += kCW * 32) {
    const uint32_t d = c.ring + kOffIdr + 32u * (uint32_t)vi;
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d), "l"(inv_delta + 8 * vi) : "memory");
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(d + 16), "l"(inv_delta + 8 * vi + 4) : "memory");
  }
  asm volatile("cp.async.commit_group;\n" ::: "memory");
}

// K1 on the input row in shared memory: x_hat = x * (1 / delta), m = max |x_hat|, s = m / 127,
// q = clamp(rint(x_hat * (127 / m)), -127, 127) (the per-token quantiser's arithmetic); x_hat is
// formed twice (for the maximum, then for the codes) rather than kept in registers.
__device__ __forceinline__ void quantize_input(Ctx& c, int K) {
  asm volatile("cp.async.wait_group 0;\n" ::: "memory");  // this thread's 1 / delta vectors
  const int nv = K >> 3;
  auto smooth8 = [&](int vi, float (&xh)[8]) {
    float x[8];
    unpack8(*reinterpret_cast<const uint4*>(c.sm + kOffX + 16 * vi), x);
    const float4 d0 = *reinterpret_cast<const float4*>(c.sm + kOffIdr + 32 * vi);
    const float4 d1 = *reinterpret_cast<const float4*>(c.sm + kOffIdr + 32 * vi + 16);
    xh[0] = __fmul_rn(x[0], d0.x);
    xh[1] = __fmul_rn(x[1], d0.y);
    xh[2] = __fmul_rn(x[2], d0.z);
    xh[3] = __fmul_rn(x[3], d0.w);
    xh[4] = __fmul_rn(x[4], d1.x);
    xh[5] = __fmul_rn(x[5], d1.y);
    xh[6] = __fmul_rn(x[6], d1.z);
    xh[7] = __fmul_rn(x[7], d1.w);
  };
  float amax = 0.0f;
  for (int vi = c.tid; vi < nv; vi += kCW * 32) {
    float xh[8];
    smooth8(vi, xh);
#pragma unroll
    for (int e = 0; e < 8; ++e) amax = fmaxf(amax, fabsf(xh[e]));
  }
  amax = warp_max(amax);
  if (c.lane == 0) c.red[c.warp] = amax;
  named_bar_sync(1, kCW * 32);
  float mx = 0.0f;
#pragma unroll
  for (int i = 0; i < kCW; ++i) mx = fmaxf(mx, c.red[i]);
  const float r = mx > 0.0f ? __fdiv_rn(127.0f, mx) : 0.0f;  // fl32(127 / m_t)
  if (c.tid == 0) *c.sx = __fdiv_rn(mx, 127.0f);             // s_t^x = fl32(m_t / 127)
  for (int vi = c.tid; vi < nv; vi += kCW * 32) {
    float xh[8];
    smooth8(vi, xh);
    int q[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) q[e] = max(-127, min(127, __float2int_rn(__fmul_rn(xh[e], r))));
    uint2 p;
    p.x = (uint32_t)(q[0] & 0xff) | ((uint32_t)(q[1] & 0xff) << 8) | ((uint32_t)(q[2] & 0xff) << 16) |
          ((uint32_t)(q[3] & 0xff) << 24);
    p.y = (uint32_t)(q[4] & 0xff) | ((uint32_t)(q[5] & 0xff) << 8) | ((uint32_t)(q[6] & 0xff) << 16) |
          ((uint32_t)(q[7] & 0xff) << 24);
    *reinterpret_cast<uint2*>(c.sm + kOffXq + 8 * vi) = p;
  }
  named_bar_sync(1, kCW * 32);
}

// This warp is done with the current slot: the last of the 8 warps refills it with the stage
// kStages ahead (the empty barrier orders every warp's reads of the slot before the copy).
__device__ __forceinline__ void release_stage(Ctx& c) {
  if (c.lane == 0) {
    mbar_arrive(c.empty0 + 8 * c.s);
    if (atomicAdd(c.slot_cnt + c.s, 1) == kCW - 1) {
      c.slot_cnt[c.s] = 0;
      atomicAdd(c.consumed, 1);
      if (mbar_wait_bounded(c.empty0 + 8 * c.s, c.ph, kWaitBudgetCycles)) {
        if (c.ahead.valid) {
          issue_stage(c.ahead, c.ring, c.s, c.full0 + 8 * c.s);
          atomicAdd(c.issued, 1);
        }
      } else {
        atomicOr(c.a->err, DEVERR_PRODUCER_WAIT);
      }
    }
  }
  cursor_next(*c.a, c.cta, c.G, c.ahead);
  if (++c.s == kStages) {
    c.s = 0;
    c.ph ^= 1u;
  }
}

// On failure, before the CTA exits: wait (bounded) for the copies of stages issued and not yet
// released (at most kStages, one per slot, so each slot's parity is unambiguous).
__device__ __forceinline__ void drain(Ctx& c) {
  if (c.tid != 0) return;
  const int done = atomicAdd(c.consumed, 0), n = atomicAdd(c.issued, 0);
  for (int i = done; i < n; ++i) {
    if (!mbar_wait_bounded(c.full0 + 8 * (uint32_t)(i % kStages), (uint32_t)((i / kStages) & 1), kWaitBudgetCycles)) {
      atomicOr(c.a->err, DEVERR_DRAIN_WAIT);
      break;
    }
  }
}

// The CTA's rows of one linear against the input row (bf16 at kOffX, or codes at kOffXq with
// scale *c.sx): out[row] in bf16, or for gate/up h[8 (grp / 2) + w] = GeGLU(gate, up).
template <bool kI8>
__device__ __forceinline__ bool linear_rows(Ctx& c, const Lin& g, const float* s_w, uint16_t* out, bool geglu) {
  float gate = 0.0f;
  const float sx = kI8 ? *c.sx : 0.0f;
#pragma unroll 1
  for (int grp = g.g0; grp < g.g1; ++grp) {
    const int row = 8 * grp + c.warp;
    const bool live = row < g.N;
    const float swr = kI8 && live ? ld_f1(s_w + row) : 0.0f;
    float f0 = 0.0f, f1 = 0.0f;
    int i0 = 0, i1 = 0;
#pragma unroll 1
    for (int k0 = 0; k0 < g.K; k0 += g.kc) {
      bool got = true;
      if (c.lane == 0) got = mbar_wait_bounded(c.full0 + 8 * c.s, c.ph, kWaitBudgetCycles);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        if (c.lane == 0) atomicOr(c.a->err, DEVERR_CONSUMER_WAIT);
        return false;
      }
      const int bytes = min(g.kc, g.K - k0) * (kI8 ? 1 : 2);
      if (live) {
        const uint32_t rb = c.ring + (uint32_t)(c.s * kSB) + (uint32_t)(c.warp * bytes);
        const int nch = bytes >> 4;
        // all of this lane's pieces of the row (at most 5: 2304 bytes / 32 lanes / 16 bytes) in flight
        // before any arithmetic
        // two pieces of the row per lane in flight at a time
        const uint32_t xb = kI8 ? c.xq + (uint32_t)k0 : c.xs + (uint32_t)(2 * k0);
        int ch = c.lane;
#pragma unroll 1
        for (; ch + 32 < nch; ch += 64) {
          const uint4 w0 = lds128(rb + 16 * ch), x0 = lds128(xb + 16 * ch);
          const uint4 w1 = lds128(rb + 16 * (ch + 32)), x1 = lds128(xb + 16 * (ch + 32));
          if constexpr (kI8) {
            i0 = __dp4a((int)w0.x, (int)x0.x, i0);
            i0 = __dp4a((int)w0.y, (int)x0.y, i0);
            i0 = __dp4a((int)w0.z, (int)x0.z, i0);
            i0 = __dp4a((int)w0.w, (int)x0.w, i0);
            i1 = __dp4a((int)w1.x, (int)x1.x, i1);
            i1 = __dp4a((int)w1.y, (int)x1.y, i1);
            i1 = __dp4a((int)w1.z, (int)x1.z, i1);
            i1 = __dp4a((int)w1.w, (int)x1.w, i1);
          } else {
            float w[8], x[8], v[8], z[8];
            unpack8(w0, w);
            unpack8(x0, x);
            unpack8(w1, v);
            unpack8(x1, z);
#pragma unroll
            for (int e = 0; e < 8; ++e) {
              f0 = fmaf(w[e], x[e], f0);
              f1 = fmaf(v[e], z[e], f1);
            }
          }
        }
        if (ch < nch) {
          const uint4 w0 = lds128(rb + 16 * ch), x0 = lds128(xb + 16 * ch);
          if constexpr (kI8) {
            i0 = __dp4a((int)w0.x, (int)x0.x, i0);
            i0 = __dp4a((int)w0.y, (int)x0.y, i0);
            i0 = __dp4a((int)w0.z, (int)x0.z, i0);
            i0 = __dp4a((int)w0.w, (int)x0.w, i0);
          } else {
            float w[8], x[8];
            unpack8(w0, w);
            unpack8(x0, x);
#pragma unroll
            for (int e = 0; e < 8; ++e) f0 = fmaf(w[e], x[e], f0);
          }
        }
      }
      __syncwarp();
      release_stage(c);
    }
    float v;
    if constexpr (kI8) {
      const int acc = warp_sum_i(i0 + i1);  // exact in any order
      v = __fmul_rn(__fmul_rn(sx, swr), __int2float_rn(acc));
    } else {
      v = warp_sum_f(f0 + f1);
    }
    if (c.lane == 0 && live) {
      if (!geglu) {
        out[row] = f32_to_bf16_bits(v);
      } else if ((grp & 1) == 0) {
        gate = v;
      } else {
        out[8 * (grp >> 1) + c.warp] = f32_to_bf16_bits(geglu_recipe(gate, v));
      }
    }
  }
  return true;
}

// ------------------------------------------------------------------------------ attention
struct RopeC {
  float w1[4], w2[4], cs[4], sn[4];
};
__device__ __forceinline__ void rope_load(RopeC& k, const float* nw, const float* cos_row, const float* sin_row,
                                          int lane) {
  const float4 cc = ld_f4(cos_row + 4 * lane);
  const float4 ss = ld_f4(sin_row + 4 * lane);
  k.cs[0] = cc.x; k.cs[1] = cc.y; k.cs[2] = cc.z; k.cs[3] = cc.w;
  k.sn[0] = ss.x; k.sn[1] = ss.y; k.sn[2] = ss.z; k.sn[3] = ss.w;
  if (nw) {
    const float4 a = ld_f4(nw + 4 * lane);
    const float4 b = ld_f4(nw + kHd / 2 + 4 * lane);
    k.w1[0] = a.x; k.w1[1] = a.y; k.w1[2] = a.z; k.w1[3] = a.w;
    k.w2[0] = b.x; k.w2[1] = b.y; k.w2[2] = b.z; k.w2[3] = b.w;
  }
}
// One head held by a warp as lane l's pairs (4l + e, 128 + 4l + e): RMSNorm (when nw) then RoPE.
__device__ __forceinline__ void rope_head(const uint16_t* src, const float* nw, const RopeC& k, float eps, int lane,
                                          float (&x1)[4], float (&x2)[4]) {
  const uint2 a = __ldcg(reinterpret_cast<const uint2*>(src + 4 * lane));
  const uint2 b = __ldcg(reinterpret_cast<const uint2*>(src + kHd / 2 + 4 * lane));
  x1[0] = bf16_lo(a.x); x1[1] = bf16_hi(a.x); x1[2] = bf16_lo(a.y); x1[3] = bf16_hi(a.y);
  x2[0] = bf16_lo(b.x); x2[1] = bf16_hi(b.x); x2[2] = bf16_lo(b.y); x2[3] = bf16_hi(b.y);
  if (nw) {
    float ss = 0.0f;
#pragma unroll
    for (int e = 0; e < 4; ++e) ss += x1[e] * x1[e] + x2[e] * x2[e];
    const float inv = 1.0f / sqrtf(warp_sum_f(ss) / (float)kHd + eps);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      x1[e] = x1[e] * inv * k.w1[e];
      x2[e] = x2[e] * inv * k.w2[e];
    }
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float y1 = x1[e] * k.cs[e] - x2[e] * k.sn[e];
    const float y2 = x2[e] * k.cs[e] + x1[e] * k.sn[e];
    x1[e] = y1;
    x2[e] = y2;
  }
}
__device__ __forceinline__ void store_bf16_head(uint16_t* dst, int lane, const float (&x1)[4], const float (&x2)[4]) {
  uint2 u1, u2;
  u1.x = (uint32_t)f32_to_bf16_bits(x1[0]) | ((uint32_t)f32_to_bf16_bits(x1[1]) << 16);
  u1.y = (uint32_t)f32_to_bf16_bits(x1[2]) | ((uint32_t)f32_to_bf16_bits(x1[3]) << 16);
  u2.x = (uint32_t)f32_to_bf16_bits(x2[0]) | ((uint32_t)f32_to_bf16_bits(x2[1]) << 16);
  u2.y = (uint32_t)f32_to_bf16_bits(x2[2]) | ((uint32_t)f32_to_bf16_bits(x2[3]) << 16);
  *reinterpret_cast<uint2*>(dst + 4 * lane) = u1;
  *reinterpret_cast<uint2*>(dst + kHd / 2 + 4 * lane) = u2;
}

// Splits of the key range per query head at this context length.
__device__ __forceinline__ int attn_splits(int len, int n_q, int G) {
  return max(1, min(min(kMegaMaxSplits, G / n_q), (len + 15) / 16));
}

// The attention phase of layer l for this CTA (a no-op for CTAs past n_q x splits).
__device__ __forceinline__ void attention(Ctx& c, const MegaLayer& Ly, int l, int pos) {
  const MegaArgs& a = *c.a;
  const int lo = Ly.window > 0 ? max(0, pos - Ly.window + 1) : 0;
  const int len = pos - lo + 1;
  const int used = attn_splits(len, a.n_q, c.G);
  if (c.cta >= a.n_q * used) return;
  const int hq = c.cta % a.n_q, r = c.cta / a.n_q, gq = a.n_q / a.n_kv, kvh = hq / gq;
  const int chunk = (len + used - 1) / used;
  const int kb = min(pos + 1, lo + r * chunk), ke = min(pos + 1, kb + chunk);
  const bool owns_new = kb < ke && ke == pos + 1;
  const size_t rs = (size_t)a.n_kv * kHd;  // cache row stride
  const uint16_t* qkv = a.qkv;
  const float* cos_row = Ly.rope_cos + (size_t)pos * (kHd / 2);
  const float* sin_row = Ly.rope_sin + (size_t)pos * (kHd / 2);
  float* qs = reinterpret_cast<float*>(c.sm + kOffQ);
  uint16_t* kn = reinterpret_cast<uint16_t*>(c.sm + kOffKn);
  uint16_t* vn = reinterpret_cast<uint16_t*>(c.sm + kOffVn);
  const bool writer = owns_new && hq % gq == 0;  // one CTA per key/value head writes the cache row
  if (c.warp == 0) {
    RopeC k;
    rope_load(k, Ly.q_norm, cos_row, sin_row, c.lane);
    float x1[4], x2[4];
    rope_head(qkv + (size_t)hq * kHd, Ly.q_norm, k, a.eps, c.lane, x1, x2);
    *reinterpret_cast<float4*>(qs + 4 * c.lane) = make_float4(x1[0] * a.scale, x1[1] * a.scale, x1[2] * a.scale,
                                                              x1[3] * a.scale);
    *reinterpret_cast<float4*>(qs + kHd / 2 + 4 * c.lane) =
        make_float4(x2[0] * a.scale, x2[1] * a.scale, x2[2] * a.scale, x2[3] * a.scale);
  } else if (c.warp == 1 && owns_new) {
    RopeC k;
    rope_load(k, Ly.k_norm, cos_row, sin_row, c.lane);
    float x1[4], x2[4];
    rope_head(qkv + (size_t)(a.n_q + kvh) * kHd, Ly.k_norm, k, a.eps, c.lane, x1, x2);
    store_bf16_head(kn, c.lane, x1, x2);
    if (writer) store_bf16_head(Ly.kc + (size_t)pos * rs + (size_t)kvh * kHd, c.lane, x1, x2);
  } else if (c.warp == 2 && owns_new) {
    const uint4 v = __ldcg(reinterpret_cast<const uint4*>(qkv + (size_t)(a.n_q + a.n_kv + kvh) * kHd) + c.lane);
    reinterpret_cast<uint4*>(vn)[c.lane] = v;
    if (writer) reinterpret_cast<uint4*>(Ly.vc + (size_t)pos * rs + (size_t)kvh * kHd)[c.lane] = v;
  }
  named_bar_sync(1, kCW * 32);

  // warp w: keys kb + w, kb + w + 8, ... in pairs (both rows' loads in flight before the math)
  float q[8];
  {
    const float4 q0 = reinterpret_cast<const float4*>(qs + 8 * c.lane)[0];
    const float4 q1 = reinterpret_cast<const float4*>(qs + 8 * c.lane)[1];
    q[0] = q0.x; q[1] = q0.y; q[2] = q0.z; q[3] = q0.w; q[4] = q1.x; q[5] = q1.y; q[6] = q1.z; q[7] = q1.w;
  }
  float m = -INFINITY, lsum = 0.0f, acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll 1
  for (int j0 = kb + c.warp; j0 < ke; j0 += 2 * kCW) {
    uint4 kr[2], vr[2];
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int j = j0 + u * kCW;
      if (j < ke) {
        if (j == pos) {
          kr[u] = reinterpret_cast<const uint4*>(kn)[c.lane];
          vr[u] = reinterpret_cast<const uint4*>(vn)[c.lane];
        } else {
          kr[u] = __ldcg(reinterpret_cast<const uint4*>(Ly.kc + (size_t)j * rs + (size_t)kvh * kHd) + c.lane);
          vr[u] = __ldcg(reinterpret_cast<const uint4*>(Ly.vc + (size_t)j * rs + (size_t)kvh * kHd) + c.lane);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < 2; ++u) {
      const int j = j0 + u * kCW;
      if (j >= ke) break;
      float kx[8];
      unpack8(kr[u], kx);
      float d = 0.0f;
#pragma unroll
      for (int e = 0; e < 8; ++e) d = fmaf(q[e], kx[e], d);
      const float sc = warp_sum_f(d);
      const float m_new = fmaxf(m, sc);
      const float corr = expf(m - m_new);  // 0 on the first key (m = -inf)
      const float p = expf(sc - m_new);
      lsum = lsum * corr + p;
      float vx[8];
      unpack8(vr[u], vx);
#pragma unroll
      for (int e = 0; e < 8; ++e) acc[e] = fmaf(p, vx[e], acc[e] * corr);
      m = m_new;
    }
  }
  float* pw = reinterpret_cast<float*>(c.sm + kOffPart) + c.warp * kPartF;
  *reinterpret_cast<float4*>(pw + 8 * c.lane) = make_float4(acc[0], acc[1], acc[2], acc[3]);
  *reinterpret_cast<float4*>(pw + 8 * c.lane + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
  if (c.lane == 0) {
    pw[kHd] = m;
    pw[kHd + 1] = lsum;
  }
  named_bar_sync(1, kCW * 32);
  if (c.warp != 0) return;
  // warp 0: the CTA's partial, then (last CTA of the head) the combination of all splits
  const float* p0 = reinterpret_cast<const float*>(c.sm + kOffPart);
  float M = -INFINITY;
#pragma unroll 1
  for (int w = 0; w < kCW; ++w) M = fmaxf(M, p0[w * kPartF + kHd]);
  float Lc = 0.0f, y[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll 1
  for (int w = 0; w < kCW; ++w) {
    const float* pg = p0 + w * kPartF;
    const float mg = pg[kHd];
    const float f = mg == -INFINITY ? 0.0f : expf(mg - M);  // warps without keys weigh nothing
    Lc += pg[kHd + 1] * f;
    const float4 x0 = reinterpret_cast<const float4*>(pg + 8 * c.lane)[0];
    const float4 x1 = reinterpret_cast<const float4*>(pg + 8 * c.lane)[1];
    y[0] = fmaf(x0.x, f, y[0]); y[1] = fmaf(x0.y, f, y[1]); y[2] = fmaf(x0.z, f, y[2]); y[3] = fmaf(x0.w, f, y[3]);
    y[4] = fmaf(x1.x, f, y[4]); y[5] = fmaf(x1.y, f, y[5]); y[6] = fmaf(x1.z, f, y[6]); y[7] = fmaf(x1.w, f, y[7]);
  }
  float* gp = a.part + ((size_t)hq * kMegaMaxSplits + r) * kPartStride;
  __stcg(reinterpret_cast<float4*>(gp + 8 * c.lane), make_float4(y[0], y[1], y[2], y[3]));
  __stcg(reinterpret_cast<float4*>(gp + 8 * c.lane + 4), make_float4(y[4], y[5], y[6], y[7]));
  if (c.lane == 0) {
    __stcg(gp + kHd, M);
    __stcg(gp + kHd + 1, Lc);
  }
  __threadfence();
  __syncwarp();
  unsigned int prev = 0;
  if (c.lane == 0) {
    __threadfence();
    prev = atomicAdd(a.sync + (size_t)a.L * 5 + (size_t)l * a.n_q + hq, 1u);
  }
  prev = __shfl_sync(0xffffffffu, prev, 0);
  if (prev != (unsigned)(used - 1)) return;
  __threadfence();
  const float* hp = a.part + (size_t)hq * kMegaMaxSplits * kPartStride;
  const float mi = c.lane < used ? __ldcg(hp + (size_t)c.lane * kPartStride + kHd) : -INFINITY;
  const float li = c.lane < used ? __ldcg(hp + (size_t)c.lane * kPartStride + kHd + 1) : 0.0f;
  const float mx = warp_max(mi);
  const float fi = mi == -INFINITY ? 0.0f : expf(mi - mx);
  const float L = warp_sum_f(li * fi);
  float z[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll 1
  for (int i = 0; i < used; ++i) {
    const float f = __shfl_sync(0xffffffffu, fi, i);
    const float* pi = hp + (size_t)i * kPartStride + 8 * c.lane;
    const float4 x0 = __ldcg(reinterpret_cast<const float4*>(pi));
    const float4 x1 = __ldcg(reinterpret_cast<const float4*>(pi) + 1);
    z[0] = fmaf(x0.x, f, z[0]); z[1] = fmaf(x0.y, f, z[1]); z[2] = fmaf(x0.z, f, z[2]); z[3] = fmaf(x0.w, f, z[3]);
    z[4] = fmaf(x1.x, f, z[4]); z[5] = fmaf(x1.y, f, z[5]); z[6] = fmaf(x1.z, f, z[6]); z[7] = fmaf(x1.w, f, z[7]);
  }
#pragma unroll
  for (int e = 0; e < 8; ++e) z[e] = z[e] / L;
  reinterpret_cast<uint4*>(a.att + (size_t)hq * kHd)[c.lane] = pack8(z);
}

// ------------------------------------------------------------------------------ the kernel
__global__ void __launch_bounds__(kThreads, 1) decode_mega_kernel(const __grid_constant__ MegaArgs a) {
  extern __shared__ uint8_t smem_raw[];
  __shared__ __align__(8) uint64_t bars[2 * kStages];
  __shared__ int s_cnt[kStages];
  __shared__ int s_issued, s_consumed;
  __shared__ float s_red[kCW];
  __shared__ int s_flag;
  __shared__ float s_sx;
  uint8_t* sm = smem_raw + ((128u - (smem_u32(smem_raw) & 127u)) & 127u);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int cta = blockIdx.x, G = gridDim.x;
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * kStages;
  if (threadIdx.x == 0) {
    for (int s = 0; s < kStages; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, kCW);
      s_cnt[s] = 0;
    }
    fence_mbar_init();
    // the first kStages stages of the weight stream
    Cursor u;
    cursor_start(a, cta, G, u);
    int n = 0;
    for (; n < kStages && u.valid; ++n) {
      issue_stage(u, smem_u32(sm), n, full0 + 8 * n);
      cursor_next(a, cta, G, u);
    }
    s_issued = n;
    s_consumed = 0;
  }
  __syncthreads();

  Ctx c;
  c.a = &a;
  c.sm = sm;
  c.ring = smem_u32(sm);
  c.full0 = full0;
  c.empty0 = empty0;
  c.slot_cnt = s_cnt;
  c.issued = &s_issued;
  c.consumed = &s_consumed;
  cursor_start(a, cta, G, c.ahead);
  for (int i = 0; i < kStages; ++i) cursor_next(a, cta, G, c.ahead);
  c.xs = c.ring + kOffX;
  c.xq = c.ring + kOffXq;
  c.red = s_red;
  c.flag = &s_flag;
  c.sx = &s_sx;
  c.cta = cta;
  c.G = G;
  c.tid = threadIdx.x;
  c.warp = warp;
  c.lane = lane;
  c.s = 0;
  c.ph = 0;
  const int pos = *a.pos;
  float* rc = a.r0;  // the residual stream as of now
  float* rn = a.r1;  // where the next residual step writes

  for (int l = 0; l < a.L; ++l) {
    const MegaLayer& Ly = a.layers[l];
    const int base = 5 * l;
    // constants of the layer's residual steps (this thread's 8 channels) and of K1, read before
    // waiting: the post-FFN / pre-attention weights, then post-attention / pre-FFN
    float wp[8], wn[8];
    auto load_w = [&](const float* p, const float* q) {
      if (p != nullptr && c.tid < (a.H >> 3)) {
        const float4 a0 = ld_f4(p + 8 * c.tid);
        const float4 a1 = ld_f4(p + 8 * c.tid + 4);
        const float4 b0 = ld_f4(q + 8 * c.tid);
        const float4 b1 = ld_f4(q + 8 * c.tid + 4);
        wp[0] = a0.x; wp[1] = a0.y; wp[2] = a0.z; wp[3] = a0.w; wp[4] = a1.x; wp[5] = a1.y; wp[6] = a1.z; wp[7] = a1.w;
        wn[0] = b0.x; wn[1] = b0.y; wn[2] = b0.z; wn[3] = b0.w; wn[4] = b1.x; wn[5] = b1.y; wn[6] = b1.z; wn[7] = b1.w;
      }
    };
    auto run_linear = [&](int j, uint16_t* out, bool geglu) -> bool {
      const Lin g = lin_of(a, Ly, l, j, cta, G);
      if (g.i8) quantize_input(c, g.K);
      return g.i8 ? linear_rows<true>(c, g, Ly.s_w[j], out, geglu) : linear_rows<false>(c, g, nullptr, out, geglu);
    };
    const bool att8 = ((a.attn_bits >> l) & 1u) != 0u, ffn8 = ((a.ffn_bits >> l) & 1u) != 0u;

    // ---- q/k/v projection (with the previous layer's post-FFN residual step)
    if (l > 0) load_w(a.layers[l - 1].ln_post_ffn, Ly.ln_in);
    if (att8) prefetch_idr(c, Ly.inv_delta[0], a.H);
    if (!wait_phase(c, l > 0 ? base - 1 : -1)) {
      drain(c);
      return;
    }
    if (l > 0) {
      residual_step(c, a.H, a.y, rc, rn, wp, wn);
      float* t = rc;
      rc = rn;
      rn = t;
    } else {
      input_copy(c, a.a0, a.H);
    }
    if (!count_phase(c, base + PH_QKV, run_linear(0, a.qkv, false))) {
      drain(c);
      return;
    }

    // ---- attention
    if (!wait_phase(c, base + PH_QKV)) {
      drain(c);
      return;
    }
    attention(c, Ly, l, pos);
    if (!count_phase(c, base + PH_ATT, true)) {
      drain(c);
      return;
    }

    // ---- o projection
    if (att8) prefetch_idr(c, Ly.inv_delta[1], a.n_q * kHd);
    if (!wait_phase(c, base + PH_ATT)) {
      drain(c);
      return;
    }
    input_copy(c, a.att, a.n_q * kHd);
    if (!count_phase(c, base + PH_O, run_linear(1, a.y, false))) {
      drain(c);
      return;
    }

    // ---- gate/up + GeGLU (with the post-attention residual step)
    load_w(Ly.ln_post_attn, Ly.ln_pre_ffn);
    if (ffn8) prefetch_idr(c, Ly.inv_delta[2], a.H);
    if (!wait_phase(c, base + PH_O)) {
      drain(c);
      return;
    }
    residual_step(c, a.H, a.y, rc, rn, wp, wn);
    {
      float* t = rc;
      rc = rn;
      rn = t;
    }
    if (!count_phase(c, base + PH_GU, run_linear(2, a.h, true))) {
      drain(c);
      return;
    }

    // ---- down
    if (ffn8) prefetch_idr(c, Ly.inv_delta[3], a.F);
    if (!wait_phase(c, base + PH_GU)) {
      drain(c);
      return;
    }
    input_copy(c, a.h, a.F);
    if (!count_phase(c, base + PH_DOWN, run_linear(3, a.y, false))) {
      drain(c);
      return;
    }
  }
}

}  // namespace

bool decode_mega_supported(int H, int F, int n_q, int n_kv, int hd, int sms) {
  if (hd != kHd || n_kv <= 0 || n_q % n_kv != 0 || n_q > 32) return false;
  if (H % 16 != 0 || H > 2048 || F % 16 != 0 || F > kMaxK || n_q * kHd > kMaxK) return false;
  return sms >= 8 * n_q;
}

w8a8_status launch_decode_mega(const MegaArgs& a, cudaStream_t st) {
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(decode_mega_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmemAlloc));
    attr_set[dev] = true;
  }
  int sms = 0, per_sm = 0;
  W8A8_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
  W8A8_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, decode_mega_kernel, kThreads, kSmemAlloc));
  W8A8_CHECK_ARG(per_sm >= 1, W8A8_ERR_UNSUPPORTED, "persistent decode kernel does not fit on an SM");
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)sms);
  cfg.blockDim = dim3(kThreads);
  cfg.dynamicSmemBytes = kSmemAlloc;
  cfg.stream = st;
  cudaLaunchAttribute at[1];
  at[0].id = cudaLaunchAttributeCooperative;  // all CTAs resident at once: they wait on each other
  at[0].val.cooperative = 1;
  cfg.attrs = at;
  cfg.numAttrs = 1;
  W8A8_CUDA(cudaLaunchKernelEx(&cfg, decode_mega_kernel, a));
  return W8A8_OK;
}

}  // namespace w8a8
