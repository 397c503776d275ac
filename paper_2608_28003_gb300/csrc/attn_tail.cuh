// Decode attention of one sequence run as the tail of its q/k/v projection (the row-owning decode
// GEMV), so that a decode step of one sequence needs no separate attention launch.
//
// The q/k/v GEMV's CTAs each write a few rows of the new q/k/v row.  When a CTA is done it takes a
// ticket (global counter, after a memory fence); the CTAs holding the last NT tickets become the
// attention CTAs.  Each of them waits (bounded) until every CTA has taken its ticket, so the whole
// q/k/v row is written, then, with the arithmetic of the decode attention kernel: applies QK-norm and
// RoPE to the new row (the CTA whose key share ends at the new position also writes its key and
// value to the cache), runs its share of the cached keys (copied into shared memory with cp.async),
// combines its warps' partials and stores one partial (m, l, o) per head in global scratch.  A second
// ticket elects the last attention CTA, which combines the NT partials per head in a fixed order and
// writes the bf16 output row, then resets both counters for the next launch.  The grid ends only after
// that, so the o projection (launched after this kernel) sees the output row.
#pragma once

#include "attn_common.cuh"

namespace w8a8 {

struct AttnTail {
  int n_q;                  // query heads (one key/value head of kAttnHd)
  int window;               // sliding window, 0 for global attention
  int max_seq;              // cache rows per sequence
  float scale, eps;         // attention scale, RMSNorm epsilon
  const int* pos;           // the new row's position (device)
  const float *q_norm, *k_norm;      // [kAttnHd] nullable (no QK-norm)
  const float *rope_cos, *rope_sin;  // [max_seq][kAttnHd / 2]
  uint16_t *kcache, *vcache;         // [max_seq][kAttnHd] bf16 (one sequence)
  uint16_t* o;              // [n_q * kAttnHd] bf16 output row
  float* part;              // [kTailCtas][n_q][kTailPartFloats] partials
  unsigned int* ctr;        // [2] tickets: zero before and after every launch
};

constexpr int kTailCtas = 8;        // attention CTAs at most
constexpr int kTailMinKeys = 16;    // keys per attention CTA, at least
constexpr int kTailTile = 32;       // cached rows per shared-memory tile
constexpr int kTailKRow = 528, kTailVRow = 512;  // padded key rows (conflict-free lane-per-key reads)
constexpr int kTailPartFloats = kAttnHd + 4;     // o[256], m, l, pad
constexpr int kTailMaxG = 4;
constexpr int kTailOffQ = 0;
constexpr int kTailOffKNew = kTailOffQ + kTailMaxG * kAttnHd * 4;
constexpr int kTailOffVNew = kTailOffKNew + kTailKRow;
constexpr int kTailOffBuf = kTailOffVNew + kTailVRow;
constexpr int kTailOffPart = kTailOffBuf + kTailTile * (kTailKRow + kTailVRow);
constexpr int kTailOffTicket = kTailOffPart + 8 * kTailPartFloats * 4;
constexpr int kTailSmem = kTailOffTicket + 16;  // bytes of shared memory the tail uses
constexpr size_t kTailScratchBytes = 256 + (size_t)kTailCtas * kTailMaxG * kTailPartFloats * 4;

// Acquire load of a global counter (sees every write made before the matching release by others).
__device__ __forceinline__ unsigned int ld_acquire_u32(const unsigned int* p) {
  unsigned int v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];\n" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Run by the 256 threads (8 warps) of a CTA that has written its q/k/v rows; `sm` is 16-byte
// aligned shared memory of kTailSmem bytes that nothing else uses now; `bar` is a named barrier
// id for these 256 threads.  Returns at once unless this CTA holds one of the last tickets.
__device__ __forceinline__ void attn_tail(const AttnTail& t, const uint16_t* qkv_row, uint8_t* sm, int bar,
                                          unsigned int* err) {
  unsigned int& s_ticket = *reinterpret_cast<unsigned int*>(sm + kTailOffTicket);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int P = (int)gridDim.x, NT = P < kTailCtas ? P : kTailCtas;
  __threadfence();           // this thread's output stores are visible device-wide ...
  named_bar_sync(bar, 256);  // ... for every thread of the CTA, before the ticket is taken
  if (tid == 0) s_ticket = atomicAdd(t.ctr, 1u);
  named_bar_sync(bar, 256);
  const unsigned int ticket = s_ticket;
  if (ticket < (unsigned int)(P - NT)) return;
  if (ticket >= (unsigned int)P) {  // counters left non-zero by a failed launch: give up loudly
    if (tid == 0) atomicOr(err, DEVERR_CONSUMER_WAIT);
    return;
  }
  const int s = (int)ticket - (P - NT);  // this attention CTA's key share
  const int G = t.n_q, KG = 8 / G;
  const int hw = warp % G, gw = warp / G;
  const int pos = *t.pos;
  const int lo = t.window > 0 ? max(0, pos - t.window + 1) : 0;
  const int len = pos - lo + 1;
  const int used = max(1, min(NT, (len + kTailMinKeys - 1) / kTailMinKeys));
  const int chunk = (len + used - 1) / used;
  const int kb = lo + s * chunk, ke = s < used ? min(pos + 1, kb + chunk) : kb;  // [kb, ke)
  const bool owns_new = s < used && ke == pos + 1;
  const int kc_end = owns_new ? pos : ke;  // cached rows [kb, kc_end), written by earlier steps
  const int ntiles = (ke - kb + kTailTile - 1) / kTailTile;
  const uint32_t sbase = smem_u32(sm);
  auto stage = [&](int tt) {
    const int j0 = kb + tt * kTailTile, n = min(kTailTile, kc_end - j0);
    const uint32_t kd = sbase + kTailOffBuf, vd = kd + kTailTile * kTailKRow;
    for (int i = tid; i < n * (kAttnHd / 8); i += 256) {
      const int jj = i >> 5, c = i & 31;
      const size_t off = (size_t)(j0 + jj) * kAttnHd + 8 * c;
      cp_async16(kd + (uint32_t)(jj * kTailKRow + 16 * c), t.kcache + off);
      cp_async16(vd + (uint32_t)(jj * kTailVRow + 16 * c), t.vcache + off);
    }
    cp_async_commit();
  };
  if (ntiles > 0) stage(0);
  const float* cos_row = t.rope_cos + (size_t)pos * (kAttnHd / 2);
  const float* sin_row = t.rope_sin + (size_t)pos * (kAttnHd / 2);
  RopeConsts qc, kc2;
  if (s < used && warp < G) load_rope_consts(qc, t.q_norm, cos_row, sin_row, lane);
  if (owns_new && warp == G) load_rope_consts(kc2, t.k_norm, cos_row, sin_row, lane);

  // every CTA has taken its ticket, so the whole q/k/v row is written (bounded wait)
  bool ok = true;
  if (tid == 0) {
    const long long t0 = clock64();
    while (ld_acquire_u32(t.ctr) < (unsigned int)P) {
      if (clock64() - t0 > kWaitBudgetCycles) {
        ok = false;
        atomicOr(err, DEVERR_CONSUMER_WAIT);
        break;
      }
    }
  }
  __syncwarp();
  ok = named_bar_all(bar, 256, ok);
  if (ok && s < used) {
    if (warp < G) {  // query head `warp`: norm, RoPE, scaled, fp32 to shared memory
      const uint16_t* src = qkv_row + (size_t)warp * kAttnHd;
      const uint2 a = __ldcg(reinterpret_cast<const uint2*>(src + 4 * lane));
      const uint2 c = __ldcg(reinterpret_cast<const uint2*>(src + kAttnHd / 2 + 4 * lane));
      float x1[4] = {bf16_lo(a.x), bf16_hi(a.x), bf16_lo(a.y), bf16_hi(a.y)};
      float x2[4] = {bf16_lo(c.x), bf16_hi(c.x), bf16_lo(c.y), bf16_hi(c.y)};
      norm_rope(x1, x2, t.q_norm != nullptr, qc, t.eps);
      float* qd = reinterpret_cast<float*>(sm + kTailOffQ) + warp * kAttnHd;
      *reinterpret_cast<float4*>(qd + 4 * lane) =
          make_float4(x1[0] * t.scale, x1[1] * t.scale, x1[2] * t.scale, x1[3] * t.scale);
      *reinterpret_cast<float4*>(qd + kAttnHd / 2 + 4 * lane) =
          make_float4(x2[0] * t.scale, x2[1] * t.scale, x2[2] * t.scale, x2[3] * t.scale);
    }
    if (owns_new && warp == G) {  // the new key: norm, RoPE, bf16, to the cache
      const uint16_t* src = qkv_row + (size_t)G * kAttnHd;
      const uint2 a = __ldcg(reinterpret_cast<const uint2*>(src + 4 * lane));
      const uint2 c = __ldcg(reinterpret_cast<const uint2*>(src + kAttnHd / 2 + 4 * lane));
      float x1[4] = {bf16_lo(a.x), bf16_hi(a.x), bf16_lo(a.y), bf16_hi(a.y)};
      float x2[4] = {bf16_lo(c.x), bf16_hi(c.x), bf16_lo(c.y), bf16_hi(c.y)};
      norm_rope(x1, x2, t.k_norm != nullptr, kc2, t.eps);
      uint2 u1, u2;
      u1.x = (uint32_t)f32_to_bf16_bits(x1[0]) | ((uint32_t)f32_to_bf16_bits(x1[1]) << 16);
      u1.y = (uint32_t)f32_to_bf16_bits(x1[2]) | ((uint32_t)f32_to_bf16_bits(x1[3]) << 16);
      u2.x = (uint32_t)f32_to_bf16_bits(x2[0]) | ((uint32_t)f32_to_bf16_bits(x2[1]) << 16);
      u2.y = (uint32_t)f32_to_bf16_bits(x2[2]) | ((uint32_t)f32_to_bf16_bits(x2[3]) << 16);
      uint16_t* kd = t.kcache + (size_t)pos * kAttnHd;
      *reinterpret_cast<uint2*>(kd + 4 * lane) = u1;
      *reinterpret_cast<uint2*>(kd + kAttnHd / 2 + 4 * lane) = u2;
      *reinterpret_cast<uint2*>(sm + kTailOffKNew + 8 * lane) = u1;
      *reinterpret_cast<uint2*>(sm + kTailOffKNew + kAttnHd + 8 * lane) = u2;
    }
    if (owns_new && warp == 7) {  // the new value: straight copy
      const uint4 v = __ldcg(reinterpret_cast<const uint4*>(qkv_row + (size_t)(G + 1) * kAttnHd) + lane);
      *reinterpret_cast<uint4*>(t.vcache + (size_t)pos * kAttnHd + 8 * lane) = v;
      *reinterpret_cast<uint4*>(sm + kTailOffVNew + 16 * lane) = v;
    }
  }
  named_bar_sync(bar, 256);

  // this warp's keys of every tile (head hw, key group gw)
  const float* qs = reinterpret_cast<const float*>(sm + kTailOffQ) + hw * kAttnHd;
  float m = -INFINITY, l = 0.0f, acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int tt = 0; tt < ntiles; ++tt) {
    cp_async_wait<0>();
    named_bar_sync(bar, 256);
    const int j0 = kb + tt * kTailTile;
    const uint8_t* kt = sm + kTailOffBuf;
    const uint8_t* vt = kt + kTailTile * kTailKRow;
    const int nt = min(kTailTile, ke - j0), per = (nt + KG - 1) / KG;
    const int wk0 = gw * per, nkw = min(per, nt - wk0);
    if (ok) attn_warp_keys(qs, kt, vt, kTailKRow, kTailVRow, sm + kTailOffKNew, sm + kTailOffVNew, j0, wk0, nkw, pos,
                           lane, m, l, acc);
    named_bar_sync(bar, 256);  // the buffer is refilled for tile tt + 1
    if (tt + 1 < ntiles) stage(tt + 1);
  }
  cp_async_wait<0>();

  // the warps of a head combine; the CTA's partial per head goes to global scratch
  float* wp = reinterpret_cast<float*>(sm + kTailOffPart) + warp * kTailPartFloats;
  *reinterpret_cast<float4*>(wp + 8 * lane) = make_float4(acc[0], acc[1], acc[2], acc[3]);
  *reinterpret_cast<float4*>(wp + 8 * lane + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
  if (lane == 0) {
    wp[kAttnHd] = m;
    wp[kAttnHd + 1] = l;
  }
  named_bar_sync(bar, 256);
  if (warp < G) {
    float M, Lc, y[8];
    attn_combine_warps(reinterpret_cast<const float*>(sm + kTailOffPart), kTailPartFloats, G, KG, warp, lane, M, Lc,
                       y);
    float* gp = t.part + ((size_t)s * kTailMaxG + warp) * kTailPartFloats;
    __stcg(reinterpret_cast<float4*>(gp + 8 * lane), make_float4(y[0], y[1], y[2], y[3]));
    __stcg(reinterpret_cast<float4*>(gp + 8 * lane + 4), make_float4(y[4], y[5], y[6], y[7]));
    if (lane == 0) {
      __stcg(gp + kAttnHd, M);
      __stcg(gp + kAttnHd + 1, Lc);
    }
  }
  __threadfence();  // the partial stores are visible before the second ticket
  named_bar_sync(bar, 256);
  if (tid == 0) s_ticket = atomicAdd(t.ctr + 1, 1u);
  named_bar_sync(bar, 256);
  if (s_ticket != (unsigned int)(NT - 1)) return;  // not the last attention CTA
  __threadfence();
  if (warp < G) {  // combine the NT partials of head `warp` in share order
    const float* in = t.part + (size_t)warp * kTailPartFloats;
    const float mi = lane < NT ? __ldcg(in + (size_t)lane * kTailMaxG * kTailPartFloats + kAttnHd) : -INFINITY;
    const float li = lane < NT ? __ldcg(in + (size_t)lane * kTailMaxG * kTailPartFloats + kAttnHd + 1) : 0.0f;
    const float mx = warp_max_f(mi);
    const float fi = mi == -INFINITY ? 0.0f : expf(mi - mx);
    const float Lsum = warp_sum_f(li * fi);
    float y[8] = {0, 0, 0, 0, 0, 0, 0, 0};
    for (int i = 0; i < NT; ++i) {
      const float f = __shfl_sync(0xffffffffu, fi, i);
      const float* pi = in + (size_t)i * kTailMaxG * kTailPartFloats + 8 * lane;
      const float4 a = __ldcg(reinterpret_cast<const float4*>(pi));
      const float4 c = __ldcg(reinterpret_cast<const float4*>(pi) + 1);
      y[0] = fmaf(a.x, f, y[0]); y[1] = fmaf(a.y, f, y[1]); y[2] = fmaf(a.z, f, y[2]); y[3] = fmaf(a.w, f, y[3]);
      y[4] = fmaf(c.x, f, y[4]); y[5] = fmaf(c.y, f, y[5]); y[6] = fmaf(c.z, f, y[6]); y[7] = fmaf(c.w, f, y[7]);
    }
    uint4 w;
    float z[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) z[e] = y[e] / Lsum;
    w.x = (uint32_t)f32_to_bf16_bits(z[0]) | ((uint32_t)f32_to_bf16_bits(z[1]) << 16);
    w.y = (uint32_t)f32_to_bf16_bits(z[2]) | ((uint32_t)f32_to_bf16_bits(z[3]) << 16);
    w.z = (uint32_t)f32_to_bf16_bits(z[4]) | ((uint32_t)f32_to_bf16_bits(z[5]) << 16);
    w.w = (uint32_t)f32_to_bf16_bits(z[6]) | ((uint32_t)f32_to_bf16_bits(z[7]) << 16);
    *reinterpret_cast<uint4*>(t.o + (size_t)warp * kAttnHd + 8 * lane) = w;
  }
  if (tid == 0) {  // every CTA has taken both tickets it will take: reset for the next launch
    t.ctr[0] = 0u;
    t.ctr[1] = 0u;
  }
}

}  // namespace w8a8
