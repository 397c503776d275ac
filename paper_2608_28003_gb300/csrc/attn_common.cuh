// Device helpers of the decode attention kernel: asynchronous row copies, warp reductions, bf16
// unpacking, the per-head RMSNorm + RoPE of the new row (lane l of a warp holds the rotate-half pairs
// (4l + e, 128 + 4l + e), e < 4), one warp's share of a key tile (scores, online softmax, values) and
// the combination of the warps' partials of a head.
#pragma once

#include "common.cuh"

namespace w8a8 {

constexpr int kAttnHd = 256;  // the head dim these kernels take

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory");
}
__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
  return v;
}
__device__ __forceinline__ float warp_max_f(float v) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
  return v;
}
__device__ __forceinline__ void unpack8_bf16(const uint4& w, float (&x)[8]) {
  x[0] = bf16_lo(w.x); x[1] = bf16_hi(w.x); x[2] = bf16_lo(w.y); x[3] = bf16_hi(w.y);
  x[4] = bf16_lo(w.z); x[5] = bf16_hi(w.z); x[6] = bf16_lo(w.w); x[7] = bf16_hi(w.w);
}

// The constants one warp needs for RMSNorm + RoPE of a head (lane l: pairs (4l + e, 128 + 4l + e)).
struct RopeConsts {
  float w1[4], w2[4], c[4], s[4];
};
__device__ __forceinline__ void load_rope_consts(RopeConsts& k, const float* nw, const float* cos_row,
                                                 const float* sin_row, int lane) {
  const float4 c = *reinterpret_cast<const float4*>(cos_row + 4 * lane);
  const float4 sn = *reinterpret_cast<const float4*>(sin_row + 4 * lane);
  k.c[0] = c.x; k.c[1] = c.y; k.c[2] = c.z; k.c[3] = c.w;
  k.s[0] = sn.x; k.s[1] = sn.y; k.s[2] = sn.z; k.s[3] = sn.w;
  if (nw) {
    const float4 a = *reinterpret_cast<const float4*>(nw + 4 * lane);
    const float4 b = *reinterpret_cast<const float4*>(nw + kAttnHd / 2 + 4 * lane);
    k.w1[0] = a.x; k.w1[1] = a.y; k.w1[2] = a.z; k.w1[3] = a.w;
    k.w2[0] = b.x; k.w2[1] = b.y; k.w2[2] = b.z; k.w2[3] = b.w;
  }
}

// RMSNorm (when has_norm) and RoPE of one head held as lane l's pairs (4l + e, 128 + 4l + e).
__device__ __forceinline__ void norm_rope(float (&x1)[4], float (&x2)[4], bool has_norm, const RopeConsts& k,
                                          float eps) {
  if (has_norm) {
    float ss = 0.0f;
#pragma unroll
    for (int e = 0; e < 4; ++e) ss += x1[e] * x1[e] + x2[e] * x2[e];
    const float inv = 1.0f / sqrtf(warp_sum_f(ss) / (float)kAttnHd + eps);
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      x1[e] = x1[e] * inv * k.w1[e];
      x2[e] = x2[e] * inv * k.w2[e];
    }
  }
#pragma unroll
  for (int e = 0; e < 4; ++e) {
    const float y1 = x1[e] * k.c[e] - x2[e] * k.s[e];
    const float y2 = x2[e] * k.c[e] + x1[e] * k.s[e];
    x1[e] = y1;
    x2[e] = y2;
  }
}


// One warp's keys [wk0, wk0 + nkw) of a tile whose key j sits at position j0 + j: scores q . k (the
// query pre-scaled, fp32 in shared memory at qs), online softmax, and the running weighted sum of
// the values (lane l holds dims 8l .. 8l+7 of acc).  Key rows at kt (kRow bytes apart) and value
// rows at vt (vRow apart), except position `pos`, whose rows are knew / vnew.  Lanes per key: 1 for
// 17-32 keys, 2 for 9-16, 4 for up to 8, so that short shares split each dot product over more
// lanes (lane = key slot * lpk + part; part p takes its own quarter / half of the 32 chunks, rotated
// so that a shared-memory phase hits 8 different bank groups).
__device__ __forceinline__ void attn_warp_keys(const float* qs, const uint8_t* kt, const uint8_t* vt, int kRow, int vRow,
                                               const uint8_t* knew, const uint8_t* vnew, int j0, int wk0, int nkw,
                                               int pos, int lane, float& m, float& l, float (&acc)[8]) {
  const int lpk = nkw > 16 ? 1 : nkw > 8 ? 2 : 4;
  const int nc = 32 / lpk, rot = lpk == 2 ? 4 : lpk == 4 ? 2 : 0;
  const int kl = lane / lpk, part = lane % lpk;
  for (int base = wk0; base < wk0 + nkw; base += 32 / lpk) {
    const int nk = min(32 / lpk, wk0 + nkw - base);  // keys of this pass
    const int j = base + kl;                          // key index within the tile
    float dsum = 0.0f;
    if (kl < nk) {
      const uint4* kr = reinterpret_cast<const uint4*>(j0 + j == pos ? knew : kt + j * kRow);
      float d[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll 8
      for (int it = 0; it < nc; ++it) {
        const int c = part * nc + ((it + part * rot) & (nc - 1));
        float kx[8];
        unpack8_bf16(kr[c], kx);
        const float4 q0 = reinterpret_cast<const float4*>(qs + 8 * c)[0];
        const float4 q1 = reinterpret_cast<const float4*>(qs + 8 * c)[1];
        float& dd = d[it & 3];
        dd = fmaf(q0.x, kx[0], dd);
        dd = fmaf(q0.y, kx[1], dd);
        dd = fmaf(q0.z, kx[2], dd);
        dd = fmaf(q0.w, kx[3], dd);
        dd = fmaf(q1.x, kx[4], dd);
        dd = fmaf(q1.y, kx[5], dd);
        dd = fmaf(q1.z, kx[6], dd);
        dd = fmaf(q1.w, kx[7], dd);
      }
      dsum = (d[0] + d[1]) + (d[2] + d[3]);
    }
    for (int o = 1; o < lpk; o <<= 1) dsum += __shfl_xor_sync(0xffffffffu, dsum, o);  // the key's parts
    const float sc = kl < nk ? dsum : -INFINITY;
    const float m_new = fmaxf(m, warp_max_f(sc));
    const float corr = expf(m - m_new);  // 0 on the first block (m = -inf)
    const float pr = kl < nk ? expf(sc - m_new) : 0.0f;
    l = l * corr + warp_sum_f(part == 0 ? pr : 0.0f);
#pragma unroll
    for (int e = 0; e < 8; ++e) acc[e] *= corr;
    for (int jj0 = 0; jj0 < nk; jj0 += 4) {  // four keys' loads in flight
      float pj[4];
      uint4 vv[4];
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const int jj = jj0 + u < nk ? jj0 + u : 0;  // past the pass: key 0 with weight 0
        pj[u] = __shfl_sync(0xffffffffu, pr, jj * lpk);
        if (jj0 + u >= nk) pj[u] = 0.0f;
        const uint8_t* vrow = (j0 + base + jj == pos) ? vnew : vt + (base + jj) * vRow;
        vv[u] = reinterpret_cast<const uint4*>(vrow)[lane];
      }
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        float vx[8];
        unpack8_bf16(vv[u], vx);
#pragma unroll
        for (int e = 0; e < 8; ++e) acc[e] = fmaf(pj[u], vx[e], acc[e]);
      }
    }
    m = m_new;
  }
}

// Warp `warp` (< G) combines the KG warps' partials of its head, stored at p0 as rows of pf floats
// [warp'][o[256], m, l] with warp' = g * G + head: the common max M, the rescaled sum Lc and lane
// l's dims 8l .. 8l+7 of the rescaled output y (empty partials, m = -inf, weigh nothing).
__device__ __forceinline__ void attn_combine_warps(const float* p0, int pf, int G, int KG, int warp, int lane,
                                                   float& M, float& Lc, float (&y)[8]) {
  M = -INFINITY;
  for (int g = 0; g < KG; ++g) M = fmaxf(M, p0[(g * G + warp) * pf + kAttnHd]);
  Lc = 0.0f;
#pragma unroll
  for (int e = 0; e < 8; ++e) y[e] = 0.0f;
  for (int g = 0; g < KG; ++g) {
    const float* pg = p0 + (g * G + warp) * pf;
    const float mg = pg[kAttnHd];
    const float f = mg == -INFINITY ? 0.0f : expf(mg - M);
    Lc += pg[kAttnHd + 1] * f;
    const float4 a = reinterpret_cast<const float4*>(pg + 8 * lane)[0];
    const float4 c = reinterpret_cast<const float4*>(pg + 8 * lane)[1];
    y[0] = fmaf(a.x, f, y[0]); y[1] = fmaf(a.y, f, y[1]); y[2] = fmaf(a.z, f, y[2]); y[3] = fmaf(a.w, f, y[3]);
    y[4] = fmaf(c.x, f, y[4]); y[5] = fmaf(c.y, f, y[5]); y[6] = fmaf(c.z, f, y[6]); y[7] = fmaf(c.w, f, y[7]);
  }
}

}  // namespace w8a8
