// Decode attention fused with QK-norm, RoPE and the KV-cache write (one new token per sequence).
//
// At decode the attention of a layer reads a few hundred cached key/value rows and one new row;
// split over separate kernels (QK-norm + RoPE, then attention with a cross-CTA combine through
// global memory) it costs several dependent round trips.  Here one launch does it all:
//  * grid (kSplits, B, n_kv x G / hpc) in clusters of kSplits CTAs along x: a cluster takes hpc of
//    the G query heads of (sequence b, key/value head kvh): all G at more than 8 sequences, one at up
//    to 8 (G times the SMs, each CTA's warps on one head); CTA r of a cluster takes an equal share of
//    the key positions; shares are at least kMinKeys long, so short contexts leave the trailing CTAs
//    idle; the first cluster of a key/value head writes the new row to the cache;
//  * before waiting for the preceding kernel (the q/k/v projection), each CTA starts copying its
//    cached key/value rows (positions before the new one, written by earlier steps) into shared
//    memory with cp.async, in tiles of 64 positions (one buffer: a share longer than a tile loads
//    the next tile after using the current one);
//  * then every working CTA applies RMSNorm (q_norm / k_norm) and RoPE to the new row with the
//    arithmetic of the prefill path (one warp per head, lane l holding the RoPE pairs
//    (4l + e, 128 + 4l + e)); the CTA whose share ends at the new position also writes its key
//    (bf16) and value to the cache and uses them from shared memory;
//  * one head per CTA (up to 8 sequences): thread t owns output dim t; per tile, half-warps score
//    the keys (the query in registers, a 16-lane shuffle sum per key), every warp takes the tile's
//    max and weights into its own shared-memory row, and thread t adds sum_j p_j v_jt; the CTA's
//    partial (m, l, o) goes to CTA 0's shared memory as one distributed shared memory store per
//    dim, and after one cluster barrier CTA 0 combines the partials, thread t its dim;
//  * G heads per CTA (more sequences): warp w handles query head w mod hpc and an even share (key
//    group w / hpc) of each tile: one, two or four lanes per key compute its dot product with the
//    scaled query (read from shared memory; key rows padded to 528 bytes, chunks rotated per lane
//    so that the lanes of a shared-memory phase hit different bank groups), then the warp updates
//    its running max, sum and output (lane l: dims 8l .. 8l+7) over its keys; the warps of a head
//    combine their partial (m, l, o) inside the CTA, each CTA stores its per-head partials into
//    CTA 0's shared memory (released by one cluster barrier), and CTA 0 combines them.
#include <cmath>

#include "attn_common.cuh"
#include "decoder_kernels.cuh"

namespace w8a8 {

namespace {

constexpr int kHd = 256;
constexpr int kSplits = 8;        // CTAs per cluster (portable cluster size)
constexpr int kMinKeys = 16;      // positions per working CTA, at least
constexpr int kTile = 64;         // positions per shared-memory tile
constexpr int kKRow = 528;        // bytes per key row in shared memory (256 bf16 + 16 bytes of padding)
constexpr int kVRow = 512;
constexpr int kBuf = kTile * (kKRow + kVRow);
constexpr int kWarps = 8;
constexpr int kPartFloats = kHd + 4;  // o[256], m, l, pad
// dynamic shared memory (about 111 KB, so that a CTA fits beside the q/k/v projection's CTAs and
// starts its copies early): queries [G][256] fp32 | new key row | new value row | one tile buffer |
// partials of the 8 warps | inbox of CTA 0 (the CTAs' per-head partials)
constexpr int kMaxG = 4;  // query heads per key/value head (the inbox is sized for this many)
constexpr int kOffQ = 0;
constexpr int kOffKNew = kOffQ + kMaxG * kHd * 4;
constexpr int kOffVNew = kOffKNew + kKRow;
constexpr int kOffBuf = kOffVNew + kVRow;
constexpr int kOffPart = kOffBuf + kBuf;
constexpr int kOffInbox = kOffPart + kWarps * kPartFloats * 4;           // CTA 0: one partial per (CTA, head)
constexpr int kSmem = kOffInbox + kSplits * kMaxG * kPartFloats * 4;

__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void st_cluster_f32(uint32_t addr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;\n" ::"r"(addr), "f"(v) : "memory");
}
__device__ __forceinline__ void st_cluster_f32x4(uint32_t addr, float a, float b, float c, float d) {
  asm volatile("st.shared::cluster.v4.f32 [%0], {%1, %2, %3, %4};\n" ::"r"(addr), "f"(a), "f"(b), "f"(c), "f"(d)
               : "memory");
}
// One query head per CTA (the cluster's head), thread t owning output dim t (256 threads, head dim
// 256).  Per key tile: half-warp h scores keys h, h + 16, ... (lane i of the half holds dims of
// chunks i and i + 16 of the key row and of the query, kept in registers; four shuffles sum the
// half); every warp then takes the tile's max and its weights p_j = e^(s_j - m) (lane i: keys i and
// i + 32) into its own shared-memory row, and thread t adds sum_j p_j v_jt to its running output.
// The CTA's (m, l, o) partial goes to CTA 0's inbox (one distributed shared memory store per dim),
// and after one cluster barrier CTA 0 combines the partials, thread t its dim.
template <typename Stage>
__device__ __forceinline__ void head_keys_one(uint8_t* sm, uint32_t sbase, Stage& stage, int kb, int ke, int ntiles,
                                              int pos, int r, int b, int hq0, const AttnShape& s,
                                              uint16_t* __restrict__ o) {
  const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
  const int half = t >> 4, l16 = lane & 15;
  const float* qs = reinterpret_cast<const float*>(sm + kOffQ);
  float4 q[4];  // dims 8 l16 .. 8 l16 + 7 and 128 + 8 l16 .. 128 + 8 l16 + 7
  q[0] = reinterpret_cast<const float4*>(qs + 8 * l16)[0];
  q[1] = reinterpret_cast<const float4*>(qs + 8 * l16)[1];
  q[2] = reinterpret_cast<const float4*>(qs + kHd / 2 + 8 * l16)[0];
  q[3] = reinterpret_cast<const float4*>(qs + kHd / 2 + 8 * l16)[1];
  float* sc = reinterpret_cast<float*>(sm + kOffPart);   // [kTile] scores of the tile
  float* pw = sc + kTile + warp * kTile;                 // this warp's weights of the tile
  float m = -INFINITY, l = 0.0f, acc = 0.0f;
  for (int ti = 0; ti < ntiles; ++ti) {
    cp_async_wait<0>();
    __syncthreads();
    const int j0 = kb + ti * kTile, nt = min(kTile, ke - j0);
    const uint8_t* kt = sm + kOffBuf;
    const uint8_t* vt = kt + kTile * kKRow;
    for (int jb = 0; jb < nt; jb += 2 * kWarps) {  // warp-uniform trip count: the shuffles below take every lane
      const int j = jb + half;
      const bool live = j < nt;
      const uint8_t* kr = j0 + j == pos ? sm + kOffKNew : kt + (live ? j : 0) * kKRow;
      const uint4 ka = reinterpret_cast<const uint4*>(kr)[l16];
      const uint4 kc = reinterpret_cast<const uint4*>(kr)[l16 + 16];
      float x[8], d0 = 0.0f, d1 = 0.0f;
      unpack8_bf16(ka, x);
      d0 = fmaf(q[0].x, x[0], d0); d0 = fmaf(q[0].y, x[1], d0); d0 = fmaf(q[0].z, x[2], d0); d0 = fmaf(q[0].w, x[3], d0);
      d0 = fmaf(q[1].x, x[4], d0); d0 = fmaf(q[1].y, x[5], d0); d0 = fmaf(q[1].z, x[6], d0); d0 = fmaf(q[1].w, x[7], d0);
      unpack8_bf16(kc, x);
      d1 = fmaf(q[2].x, x[0], d1); d1 = fmaf(q[2].y, x[1], d1); d1 = fmaf(q[2].z, x[2], d1); d1 = fmaf(q[2].w, x[3], d1);
      d1 = fmaf(q[3].x, x[4], d1); d1 = fmaf(q[3].y, x[5], d1); d1 = fmaf(q[3].z, x[6], d1); d1 = fmaf(q[3].w, x[7], d1);
      float dsum = d0 + d1;
#pragma unroll
      for (int of = 8; of > 0; of >>= 1) dsum += __shfl_xor_sync(0xffffffffu, dsum, of);  // within the half
      if (live && l16 == 0) sc[j] = dsum;
    }
    __syncthreads();
    const float s0 = lane < nt ? sc[lane] : -INFINITY, s1 = lane + 32 < nt ? sc[lane + 32] : -INFINITY;
    const float m_new = fmaxf(m, warp_max_f(fmaxf(s0, s1)));
    const float corr = expf(m - m_new);  // 0 on the first tile (m = -inf)
    const float p0 = lane < nt ? expf(s0 - m_new) : 0.0f, p1 = lane + 32 < nt ? expf(s1 - m_new) : 0.0f;
    pw[lane] = p0;
    pw[lane + 32] = p1;
    l = l * corr + warp_sum_f(p0 + p1);
    m = m_new;
    __syncwarp();
    float a4[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    int j = 0;
    for (; j + 4 <= nt; j += 4) {
#pragma unroll
      for (int u = 0; u < 4; ++u) {
        const uint8_t* vr = j0 + j + u == pos ? sm + kOffVNew : vt + (j + u) * kVRow;
        a4[u] = fmaf(pw[j + u], bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(vr)[t]), a4[u]);
      }
    }
    for (; j < nt; ++j) {
      const uint8_t* vr = j0 + j == pos ? sm + kOffVNew : vt + j * kVRow;
      a4[0] = fmaf(pw[j], bf16_bits_to_f32(reinterpret_cast<const uint16_t*>(vr)[t]), a4[0]);
    }
    acc = fmaf(acc, corr, (a4[0] + a4[1]) + (a4[2] + a4[3]));
    __syncthreads();  // the buffer, the scores and the weights are reused by the next tile
    if (ti + 1 < ntiles) stage(ti + 1);
  }
  const uint32_t dst = map_to_rank(sbase + kOffInbox + (uint32_t)(r * kMaxG * kPartFloats * 4), 0);
  st_cluster_f32(dst + 4 * t, acc);
  if (t == 0) {
    st_cluster_f32(dst + kHd * 4, m);
    st_cluster_f32(dst + (kHd + 1) * 4, l);
  }
  cluster_sync_all();  // release the pushes / acquire them in CTA 0
  if (r != 0) return;
  const float* in = reinterpret_cast<const float*>(sm + kOffInbox);
  float mr[kSplits], M = -INFINITY;
#pragma unroll
  for (int i = 0; i < kSplits; ++i) {
    mr[i] = in[i * kMaxG * kPartFloats + kHd];
    M = fmaxf(M, mr[i]);
  }
  float L = 0.0f, y = 0.0f;
#pragma unroll
  for (int i = 0; i < kSplits; ++i) {
    const float f = mr[i] == -INFINITY ? 0.0f : expf(mr[i] - M);
    L = fmaf(in[i * kMaxG * kPartFloats + kHd + 1], f, L);
    y = fmaf(in[i * kMaxG * kPartFloats + t], f, y);
  }
  o[(size_t)b * (s.n_q * kHd) + (size_t)hq0 * kHd + t] = f32_to_bf16_bits(y / L);
}

__global__ void __cluster_dims__(kSplits, 1, 1) __launch_bounds__(kWarps * 32)
    attn_decode_kernel(const uint16_t* __restrict__ qkv, AttnShape s, const int* __restrict__ pos0,
                       const float* __restrict__ qn, const float* __restrict__ kn, float eps,
                       const float* __restrict__ rope_cos, const float* __restrict__ rope_sin,
                       uint16_t* __restrict__ kcache, uint16_t* __restrict__ vcache, uint16_t* __restrict__ o,
                       int hpc) {
  extern __shared__ __align__(16) uint8_t sm[];
  pdl_trigger();
  // hpc query heads per cluster (1, or all G heads of a key/value head): blockIdx.z picks the
  // key/value head and, with hpc < G, which hpc of its query heads this cluster takes
  const int G = s.n_q / s.n_kv, KG = kWarps / hpc;  // heads per key/value head; key groups per tile
  const int r = blockIdx.x, b = blockIdx.y, kvh = blockIdx.z / (G / hpc);
  const int hq0 = kvh * G + (blockIdx.z % (G / hpc)) * hpc;  // this cluster's first query head
  const bool writes_cache = hq0 == kvh * G;  // the first cluster of a key/value head stores its new row
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int hw = warp % hpc, gw = warp / hpc;     // this warp's head (within the cluster's) and key group
  // The position was set before this launch's chain began, and cached rows before it were
  // written by earlier launches: both may be read before waiting for the preceding kernel.
  const int pos = *pos0;
  const int lo = s.window > 0 ? max(0, pos - s.window + 1) : 0;
  const int len = pos - lo + 1;
  const int used = max(1, min(kSplits, (len + kMinKeys - 1) / kMinKeys));
  const int chunk = (len + used - 1) / used;
  const int kb = lo + r * chunk, ke = r < used ? min(pos + 1, kb + chunk) : kb;  // [kb, ke)
  const bool owns_new = r < used && ke == pos + 1;
  const int kc_end = owns_new ? pos : ke;  // cached rows [kb, kc_end)
  const int ntiles = (ke - kb + kTile - 1) / kTile;
  const size_t row_stride = (size_t)s.n_kv * kHd;
  const size_t seq_base = (size_t)b * s.max_seq * row_stride + (size_t)kvh * kHd;
  const uint32_t sbase = smem_u32(sm);

  auto stage = [&](int t) {  // cached rows of tile t into the buffer
    const int j0 = kb + t * kTile, n = min(kTile, kc_end - j0);
    const uint32_t kd = sbase + kOffBuf, vd = kd + kTile * kKRow;
    for (int i = threadIdx.x; i < n * (kHd / 8); i += kWarps * 32) {
      const int jj = i >> 5, c = i & 31;
      const size_t off = seq_base + (size_t)(j0 + jj) * row_stride + 8 * c;
      cp_async16(kd + (uint32_t)(jj * kKRow + 16 * c), kcache + off);
      cp_async16(vd + (uint32_t)(jj * kVRow + 16 * c), vcache + off);
    }
    cp_async_commit();
  };
  if (ntiles > 0) stage(0);
  // norm weights and the RoPE row of this position: constants, read before the wait as well
  const float* cos_row = rope_cos + (size_t)pos * (kHd / 2);
  const float* sin_row = rope_sin + (size_t)pos * (kHd / 2);
  const int kwarp = hpc;  // the warp that rotates the new key (hpc < 8 warps)
  RopeConsts qc, kc2;
  if (r < used && warp < hpc) load_rope_consts(qc, qn, cos_row, sin_row, lane);
  if (owns_new && warp == kwarp) load_rope_consts(kc2, kn, cos_row, sin_row, lane);

  pdl_wait();
  // ---- the new row: q heads (scaled, fp32, to shared memory), and k / v for the owning CTA
  const int qkv_dim = (s.n_q + 2 * s.n_kv) * kHd;
  const uint16_t* src_row = qkv + (size_t)b * qkv_dim;
  if (r < used) {
    if (warp < hpc) {
      const uint16_t* src = src_row + (size_t)(hq0 + warp) * kHd;
      const uint2 a = *reinterpret_cast<const uint2*>(src + 4 * lane);
      const uint2 c = *reinterpret_cast<const uint2*>(src + kHd / 2 + 4 * lane);
      float x1[4] = {bf16_lo(a.x), bf16_hi(a.x), bf16_lo(a.y), bf16_hi(a.y)};
      float x2[4] = {bf16_lo(c.x), bf16_hi(c.x), bf16_lo(c.y), bf16_hi(c.y)};
      norm_rope(x1, x2, qn != nullptr, qc, eps);
      float* qd = reinterpret_cast<float*>(sm + kOffQ) + warp * kHd;
      *reinterpret_cast<float4*>(qd + 4 * lane) = make_float4(x1[0] * s.scale, x1[1] * s.scale, x1[2] * s.scale,
                                                              x1[3] * s.scale);
      *reinterpret_cast<float4*>(qd + kHd / 2 + 4 * lane) =
          make_float4(x2[0] * s.scale, x2[1] * s.scale, x2[2] * s.scale, x2[3] * s.scale);
    }
    if (owns_new && warp == kwarp) {  // key head kvh
      const uint16_t* src = src_row + (size_t)(s.n_q + kvh) * kHd;
      const uint2 a = *reinterpret_cast<const uint2*>(src + 4 * lane);
      const uint2 c = *reinterpret_cast<const uint2*>(src + kHd / 2 + 4 * lane);
      float x1[4] = {bf16_lo(a.x), bf16_hi(a.x), bf16_lo(a.y), bf16_hi(a.y)};
      float x2[4] = {bf16_lo(c.x), bf16_hi(c.x), bf16_lo(c.y), bf16_hi(c.y)};
      norm_rope(x1, x2, kn != nullptr, kc2, eps);
      uint2 u1, u2;
      u1.x = (uint32_t)f32_to_bf16_bits(x1[0]) | ((uint32_t)f32_to_bf16_bits(x1[1]) << 16);
      u1.y = (uint32_t)f32_to_bf16_bits(x1[2]) | ((uint32_t)f32_to_bf16_bits(x1[3]) << 16);
      u2.x = (uint32_t)f32_to_bf16_bits(x2[0]) | ((uint32_t)f32_to_bf16_bits(x2[1]) << 16);
      u2.y = (uint32_t)f32_to_bf16_bits(x2[2]) | ((uint32_t)f32_to_bf16_bits(x2[3]) << 16);
      if (writes_cache) {
        uint16_t* kd = kcache + seq_base + (size_t)pos * row_stride;
        *reinterpret_cast<uint2*>(kd + 4 * lane) = u1;
        *reinterpret_cast<uint2*>(kd + kHd / 2 + 4 * lane) = u2;
      }
      *reinterpret_cast<uint2*>(sm + kOffKNew + 8 * lane) = u1;
      *reinterpret_cast<uint2*>(sm + kOffKNew + kHd + 8 * lane) = u2;
    }
    if (owns_new && warp == kWarps - 1) {  // value head kvh: straight copy
      const uint16_t* src = src_row + (size_t)(s.n_q + s.n_kv + kvh) * kHd;
      const uint4 v = *reinterpret_cast<const uint4*>(src + 8 * lane);
      if (writes_cache) *reinterpret_cast<uint4*>(vcache + seq_base + (size_t)pos * row_stride + 8 * lane) = v;
      *reinterpret_cast<uint4*>(sm + kOffVNew + 16 * lane) = v;
    }
  }
  __syncthreads();

  if (hpc == 1) {  // one head per cluster: see head_keys_one
    head_keys_one(sm, sbase, stage, kb, ke, ntiles, pos, r, b, hq0, s, o);
    return;
  }

  // ---- this warp's keys of every tile
  const float* qs = reinterpret_cast<const float*>(sm + kOffQ) + hw * kHd;
  float m = -INFINITY, l = 0.0f, acc[8] = {0, 0, 0, 0, 0, 0, 0, 0};
  for (int t = 0; t < ntiles; ++t) {
    cp_async_wait<0>();
    __syncthreads();
    const int j0 = kb + t * kTile;
    const uint8_t* kt = sm + kOffBuf;
    const uint8_t* vt = kt + kTile * kKRow;
    // this warp's keys of the tile: an even share of the tile among the KG warps of its head
    const int nt = min(kTile, ke - j0), per = (nt + KG - 1) / KG;
    const int wk0 = gw * per, nkw = min(per, nt - wk0);
    attn_warp_keys(qs, kt, vt, kKRow, kVRow, sm + kOffKNew, sm + kOffVNew, j0, wk0, nkw, pos, lane, m, l, acc);
    __syncthreads();  // the buffer is refilled for tile t + 1
    if (t + 1 < ntiles) stage(t + 1);
  }

  // ---- partials: the warps of a head combine inside the CTA, the CTA pushes the result into CTA
  // 0's inbox (distributed shared memory stores), and CTA 0 combines the inbox after one barrier
  float* part = reinterpret_cast<float*>(sm + kOffPart) + warp * kPartFloats;
  *reinterpret_cast<float4*>(part + 8 * lane) = make_float4(acc[0], acc[1], acc[2], acc[3]);
  *reinterpret_cast<float4*>(part + 8 * lane + 4) = make_float4(acc[4], acc[5], acc[6], acc[7]);
  if (lane == 0) {
    part[kHd] = m;
    part[kHd + 1] = l;
  }
  __syncthreads();
  if (warp < hpc) {
    float M, Lc, y[8];
    attn_combine_warps(reinterpret_cast<const float*>(sm + kOffPart), kPartFloats, hpc, KG, warp, lane, M, Lc, y);
    const uint32_t dst = map_to_rank(sbase + kOffInbox + (uint32_t)((r * kMaxG + warp) * kPartFloats * 4), 0);
    st_cluster_f32x4(dst + 32 * lane, y[0], y[1], y[2], y[3]);
    st_cluster_f32x4(dst + 32 * lane + 16, y[4], y[5], y[6], y[7]);
    if (lane == 0) {
      st_cluster_f32(dst + kHd * 4, M);
      st_cluster_f32(dst + (kHd + 1) * 4, Lc);
    }
  }
  cluster_sync_all();  // release the pushes / acquire them in CTA 0
  if (r == 0 && warp < hpc) {
    const float* in = reinterpret_cast<const float*>(sm + kOffInbox);
    const float mi = lane < kSplits ? in[(lane * kMaxG + warp) * kPartFloats + kHd] : -INFINITY;
    const float li = lane < kSplits ? in[(lane * kMaxG + warp) * kPartFloats + kHd + 1] : 0.0f;
    const float mx = warp_max_f(mi);
    const float fi = mi == -INFINITY ? 0.0f : expf(mi - mx);
    const float L = warp_sum_f(li * fi);
    float y[8] = {0, 0, 0, 0, 0, 0, 0, 0};
#pragma unroll
    for (int i = 0; i < kSplits; ++i) {
      const float f = __shfl_sync(0xffffffffu, fi, i);
      const float* pi = in + (i * kMaxG + warp) * kPartFloats + 8 * lane;
      const float4 a = reinterpret_cast<const float4*>(pi)[0];
      const float4 c = reinterpret_cast<const float4*>(pi)[1];
      y[0] = fmaf(a.x, f, y[0]); y[1] = fmaf(a.y, f, y[1]); y[2] = fmaf(a.z, f, y[2]); y[3] = fmaf(a.w, f, y[3]);
      y[4] = fmaf(c.x, f, y[4]); y[5] = fmaf(c.y, f, y[5]); y[6] = fmaf(c.z, f, y[6]); y[7] = fmaf(c.w, f, y[7]);
    }
    uint4 w;
    float z[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) z[e] = y[e] / L;
    w.x = (uint32_t)f32_to_bf16_bits(z[0]) | ((uint32_t)f32_to_bf16_bits(z[1]) << 16);
    w.y = (uint32_t)f32_to_bf16_bits(z[2]) | ((uint32_t)f32_to_bf16_bits(z[3]) << 16);
    w.z = (uint32_t)f32_to_bf16_bits(z[4]) | ((uint32_t)f32_to_bf16_bits(z[5]) << 16);
    w.w = (uint32_t)f32_to_bf16_bits(z[6]) | ((uint32_t)f32_to_bf16_bits(z[7]) << 16);
    *reinterpret_cast<uint4*>(o + (size_t)b * (s.n_q * kHd) + (size_t)(hq0 + warp) * kHd + 8 * lane) = w;
  }
}

}  // namespace

bool attn_decode_supported(const AttnShape& s) {
  if (s.T != 1 || s.hd != kHd || s.n_kv <= 0 || s.n_q % s.n_kv != 0) return false;
  const int G = s.n_q / s.n_kv;
  return G == 2 || G == 4;
}

w8a8_status launch_attn_decode(const uint16_t* qkv, const AttnShape& s, const int* pos0, const float* qn,
                               const float* kn, float eps, const float* rope_cos, const float* rope_sin,
                               uint16_t* kcache, uint16_t* vcache, uint16_t* o, cudaStream_t st) {
  if (s.B == 0) return W8A8_OK;
  W8A8_CHECK_ARG(attn_decode_supported(s), W8A8_ERR_SHAPE,
                 "decode attention: needs one token per sequence, head_dim 256 and 2 or 4 query heads per kv head");
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(attn_decode_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kSmem));
    attr_set[dev] = true;
  }
  // Few sequences: one cluster per query head (G times the SMs, every CTA's warps on one head, the
  // cached rows read once per head); many: one cluster per key/value head (its G heads share the rows).
  const int G = s.n_q / s.n_kv, hpc = s.B <= 8 ? 1 : G;
  W8A8_CUDA(launch_pdl(attn_decode_kernel, dim3(kSplits, s.B, s.n_kv * (G / hpc)), dim3(kWarps * 32), (size_t)kSmem,
                       st, qkv, s, pos0, qn, kn, eps, rope_cos, rope_sin, kcache, vcache, o, hpc));
  return W8A8_OK;
}

}  // namespace w8a8
