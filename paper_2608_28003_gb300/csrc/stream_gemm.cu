// Weight-streaming GEMM for decode-sized token counts on the m16n8k16 tensor-core MMA.
//
// Computes acc_ti = sum_j X_tj * W_ij for W [N, K] (row = output channel) and X [M, K]: the INT8
// sum of Eq. gemm-final on the W8A8 path, the bf16 pass-through of the FFN section otherwise,
// followed by the calling layer's epilogue.  Decode is HBM-bound on W, so the kernel is built
// around moving W at full bandwidth:
//
//  * Persistent grid, two CTAs per SM up to four token blocks (32 tokens), one beyond: the second
//    CTA's warps hide the first one's MMA and widening latencies (W8A8 lm_head at 16 tokens 119 ->
//    88 us, at 32 tokens 170 -> 131 us, the latter with a few spilled registers); 1 producer warp
//    + 8 consumer warps each.  The work is the list
//    of units (token group z, 128-row weight group g, k chunk of 64..256 bytes per row), ordered
//    z-major, then g, then k; CTA c takes the contiguous range [c U / P, (c+1) U / P), so every
//    CTA streams the same number of bytes (stream-K style balance, no wave tail); the chunk
//    shrinks for small layers so that there are at least as many units as SMs.
//  * One producer thread loads each unit with 2-D TMA (cp.async.bulk.tensor): 128-byte-wide boxes
//    of 128 weight rows and of the unit's token rows of X, 128-byte swizzled, zero-filled outside
//    the tensors, into a ring of shared-memory stages guarded by mbarriers; consumers release a
//    stage through a second mbarrier.
//  * Consumer warp w owns tile rows 16w .. 16w+15 of every unit.  Lane 4g + t loads k = 16t .. 16t+15
//    (of each 64-wide step) of MMA rows g and g+8 and of token g, and feeds MMA j (j = 0..3) the
//    lane's k = 16t+4j .. 16t+4j+3 on both operands, a k permutation that a dot product does not
//    see.  MMA row g reads tile row perm(g): the identity for bf16, and for INT8 (lanes read 16 of
//    each row's 128 swizzled bytes) the pairing (2p, 2p+1) -> (p, p+4), so the two rows a phase of
//    8 lanes touches use opposite halves of the banks.
//  * W8A8 path: INT8 codes are widened to fp16 in registers (exact); X holds fp16 codes.  Each
//    product of codes is an integer below 2^14 and any partial sum of at most 1024 of them stays
//    below 2^24, where fp32 is exact, so the fp32 accumulator is folded into INT32 every 16 steps
//    (1024 k) and the INT32 result is exact in any summation order.
//  * A (z, g) whose k range spans several CTAs is finished by the last CTA to arrive: each
//    contributor writes its partial tile, bumps a counter (no waiting), and the last one sums the
//    partials in CTA order (exact for INT32; a fixed order for fp32) and runs the epilogue.
//  * Every mbarrier wait is bounded: on timeout the kernel sets a bit in the workspace's error
//    word, stops waiting, lets its own copies in flight land (again bounded) and returns.
#include <algorithm>

#include "stream_gemm.cuh"
#include "tmap.cuh"

namespace w8a8 {

namespace {

constexpr int kTileCounterSlots = 8192;                      // uint32 slots at workspace offset 0
constexpr size_t kGridCounterOffset = 8192 * 4;              // one uint32
constexpr size_t kTopKeysOffset = 40960;                     // uint64 keys
constexpr int kMaxTopKeys = (W8A8_WS_RESERVED - 40960) / 8;  // 3072
constexpr int kConsumerWarps = 8;
constexpr int kThreads = (kConsumerWarps + 1) * 32;
constexpr int kSmemLimit = 227 * 1024;   // shared memory per SM available to CTAs
constexpr int kStaticReserve = 8192;     // static shared memory of the kernel (barrier flags, top-1 keys)
constexpr int kBox = 16384;  // one weight box: 128 rows x 128 bytes

template <bool kInt8>
struct Geo {
  static constexpr int EB = kInt8 ? 1 : 2;           // weight element bytes
  static constexpr int KCMAX = kInt8 ? 256 : 128;    // stage capacity in k elements (2 weight boxes)
  static constexpr int BOXK = 128 / EB;              // k elements per weight box
};

__host__ __device__ constexpr int stage_bytes_for(bool int8, int tok) {
  // 2 weight boxes + (KCMAX / 64) token boxes of TOK rows x 128 bytes, all 1024-byte aligned
  return 2 * kBox + (int8 ? 4 : 2) * tok * 128;
}

__device__ __forceinline__ uint32_t u4c(const uint4& v, int c) {
  return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

// tile row read by MMA row g (0..7)
template <bool kInt8>
__device__ __forceinline__ int row_perm(int g) {
  return kInt8 ? ((g >> 1) | ((g & 1) << 2)) : g;
}

// CTAs per SM: two for up to 16 tokens (registers allow it), else one.
template <int NB>
struct Cps {
  static constexpr int value = NB <= 4 ? 2 : 1;
};

template <bool kInt8, int NB, int STEPS>
__global__ void __launch_bounds__(kThreads, Cps<NB>::value)
    stream_gemm_kernel(const __grid_constant__ CUtensorMap tmW, const __grid_constant__ CUtensorMap tmX,
                       const StreamArgs a) {
  using GG = Geo<kInt8>;
  constexpr int TOK = 8 * NB;
  constexpr int BOXK = GG::BOXK;
  constexpr int KC = STEPS * 64;  // k elements per unit
  constexpr int CH = NB >= 4 ? 1 : 4 / NB;  // independent accumulator chains per token block
  constexpr int XBOX = TOK * 128;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ int s_flag;
  __shared__ unsigned long long s_best[kConsumerWarps][TOK];  // top-1: per-warp best key per token slot

  const StreamPlan& p = a.p;
  const int S = p.stages, SB = p.stage_bytes;
  // 128-byte swizzle repeats every 1024 bytes: align the ring to 1024
  const uint32_t raw_u32 = smem_u32(smem_raw);
  const uint32_t ring = (raw_u32 + 1023u) & ~1023u;
  uint64_t* full = reinterpret_cast<uint64_t*>(smem_raw + (ring - raw_u32) + (size_t)S * SB);
  uint64_t* empty = full + S;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.G, C = p.C, Z = p.Z;
  const long long U = (long long)Z * G * C;
  const int P = gridDim.x, cta = blockIdx.x;
  // Unit range of this CTA: whole (z, g) groups when there are at least as many groups as CTAs
  // (no group is split, no partial tiles), else an even split of the units (stream-K).
  const long long ZG = (long long)Z * G;
  const long long u0 = p.whole ? (long long)cta * ZG / P * C : (long long)cta * U / P;
  const long long u1 = p.whole ? (long long)(cta + 1) * ZG / P * C : (long long)(cta + 1) * U / P;
  auto cta_of = [&](long long u) -> int { return (int)(((u + 1) * P + U - 1) / U - 1); };

  pdl_trigger();
  if (threadIdx.x == kConsumerWarps * 32) {  // the producer thread: fetch the tensor maps before the first copy needs them
    prefetch_tmap(&tmW);
    prefetch_tmap(&tmX);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(full + s), 1);
      mbar_init(smem_u32(empty + s), kConsumerWarps);
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (u0 >= u1) {
    pdl_wait();
    return;
  }

  // ------------------------------------------------------------------------ producer thread
  if (warp == kConsumerWarps) {
    if (lane != 0) return;
    constexpr int nw = KC / BOXK, nx = KC / 64;
    const uint32_t tx = (uint32_t)(nw * kBox + nx * XBOX);
    bool ok = true;
    long long it = 0;
    // The weights of the first stages do not depend on the preceding kernel: request them before
    // waiting for it, then add the token rows of X to the same stages.
    const long long npre = (long long)S < u1 - u0 ? (long long)S : u1 - u0;
    for (; it < npre; ++it) {
      const long long u = u0 + it;
      const int zg = (int)(u / C), ch = (int)(u % C);
      const int g = zg % G;
      const uint32_t bar = smem_u32(full + (int)it);
      mbar_arrive_expect_tx(bar, tx);
      for (int b = 0; b < nw; ++b)
        tma_load_2d(ring + (uint32_t)it * SB + b * kBox, &tmW, ch * KC + b * BOXK, g * 128, bar);
    }
    pdl_wait();
    for (long long j = 0; j < npre; ++j) {
      const long long u = u0 + j;
      const int zg = (int)(u / C), ch = (int)(u % C);
      const int z = zg / G;
      const uint32_t bar = smem_u32(full + (int)j);
      for (int b = 0; b < nx; ++b)
        tma_load_2d(ring + (uint32_t)j * SB + 2 * kBox + b * XBOX, &tmX, ch * KC + b * 64, z * TOK, bar);
    }
    for (long long u = u0 + npre; u < u1; ++u, ++it) {
      const int s = (int)(it % S);
      const uint32_t ph = (uint32_t)((it / S) & 1);
      if (!mbar_wait_bounded(smem_u32(empty + s), ph ^ 1u, kWaitBudgetCycles)) {
        ok = false;
        break;
      }
      const int zg = (int)(u / C), ch = (int)(u % C);
      const int z = zg / G, g = zg % G;
      const uint32_t bar = smem_u32(full + s);
      const uint32_t sb = ring + (uint32_t)s * SB;
      mbar_arrive_expect_tx(bar, tx);
      for (int b = 0; b < nw; ++b) tma_load_2d(sb + b * kBox, &tmW, ch * KC + b * BOXK, g * 128, bar);
      for (int b = 0; b < nx; ++b) tma_load_2d(sb + 2 * kBox + b * XBOX, &tmX, ch * KC + b * 64, z * TOK, bar);
    }
    if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
    // Let the copies of the last stages land before this CTA can exit (bounded).
    for (long long j = it > S ? it - S : 0; j < it; ++j) {
      if (!mbar_wait_bounded(smem_u32(full + (int)(j % S)), (uint32_t)((j / S) & 1), kWaitBudgetCycles)) {
        atomicOr(a.err, DEVERR_DRAIN_WAIT);
        break;
      }
    }
    return;
  }

  // ----------------------------------------------------------------------- consumer warps
  pdl_wait();
  const int w = warp;
  const int gl = lane >> 2, t = lane & 3;
  const int pr = row_perm<kInt8>(gl);  // tile row (within 16) of MMA row gl; MMA row gl+8 -> pr+8
  float acc[CH][NB][4];
  int iacc[NB][4];
  int since = 0;
  bool ok = true;
  // top-1: the warp's best key per token slot of token group best_z (in s_best), published with
  // one atomicMax per token when the token group changes and at the end
  int best_z = -1;

  auto zero_acc = [&]() {
#pragma unroll
    for (int c = 0; c < CH; ++c)
#pragma unroll
      for (int nb = 0; nb < NB; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) acc[c][nb][e] = 0.0f;
#pragma unroll
    for (int nb = 0; nb < NB; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) iacc[nb][e] = 0;
    since = 0;
  };

  auto publish_top = [&]() {
    if (best_z < 0) return;
    __syncwarp();
    for (int i = lane; i < TOK; i += 32) {
      const int tk = best_z * TOK + i;
      const unsigned long long k = s_best[w][i];
      if (tk < a.M && k != 0ull) atomicMax(a.top_keys + tk, k);
    }
    __syncwarp();
    best_z = -1;
  };

  // dequantised (or bf16-path) fp32 value of an accumulator, before the bias
  auto value_f32 = [&](uint32_t v, int i, int tk) -> float {
    if constexpr (kInt8) {
      const float sc = __fmul_rn(a.s_x[tk], a.s_w[i]);  // s_t^x * s_i^W
      return __fmul_rn(sc, __int2float_rn((int)v));
    } else {
      return __uint_as_float(v);
    }
  };

  const bool want_top = a.kind == EPI_F32 && a.top1 != nullptr;
  auto epilogue = [&](int z, int g, uint32_t (&v)[NB][4]) {
    const int ra = g * 128 + 16 * w + pr, rb = ra + 8;
    if (want_top && z != best_z) {
      publish_top();
      best_z = z;
      for (int i = lane; i < TOK; i += 32) s_best[w][i] = 0ull;
      __syncwarp();
    }
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        unsigned long long best = 0ull;
        const int tk = z * TOK + nb * 8 + 2 * t + h;
        if (tk >= a.M) {
        } else if (a.kind == EPI_GEGLU) {
          if (rb >= a.N) continue;
          float gv = value_f32(v[nb][h], ra, tk), uv = value_f32(v[nb][2 + h], rb, tk);
          if (a.bias) {
            gv = __fadd_rn(gv, a.bias[ra]);
            uv = __fadd_rn(uv, a.bias[rb]);
          }
          if constexpr (kInt8) {
            if (a.acc_dbg) {
              a.acc_dbg[(size_t)tk * a.N + ra] = (int)v[nb][h];
              a.acc_dbg[(size_t)tk * a.N + rb] = (int)v[nb][2 + h];
            }
          }
          a.y[(size_t)tk * (a.N >> 1) + ((g * 128 + 16 * w) >> 1) + pr] = f32_to_bf16_bits(geglu_recipe(gv, uv));
        } else {
#pragma unroll
          for (int side = 0; side < 2; ++side) {
            const int i = side ? rb : ra;
            if (i >= a.N) continue;
            const uint32_t raw = v[nb][2 * side + h];
            float y = value_f32(raw, i, tk);
            if (a.bias) y = __fadd_rn(y, a.bias[i]);
            if constexpr (kInt8) {
              if (a.acc_dbg) a.acc_dbg[(size_t)tk * a.N + i] = (int)raw;
            }
            if (a.kind == EPI_BF16) {
              a.y[(size_t)tk * a.N + i] = f32_to_bf16_bits(y);
            } else {
              if (a.logits) a.logits[(size_t)tk * a.N + i] = y;
              const unsigned long long key =
                  ((unsigned long long)float_order_key(y) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)i);
              best = key > best ? key : best;
            }
          }
        }
        if (want_top) {  // max over the 8 row pairs (lanes with equal t)
#pragma unroll
          for (int o = 4; o < 32; o <<= 1) {
            const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
            best = other > best ? other : best;
          }
          if (gl == 0 && best > s_best[w][nb * 8 + 2 * t + h]) s_best[w][nb * 8 + 2 * t + h] = best;
        }
      }
    }
  };

  auto flush = [&](int zg, int chf, int chl) {
    uint32_t v[NB][4];
#pragma unroll
    for (int nb = 0; nb < NB; ++nb)
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        if constexpr (kInt8) {
          int sum = iacc[nb][e];
#pragma unroll
          for (int c = 0; c < CH; ++c) sum += __float2int_rn(acc[c][nb][e]);
          v[nb][e] = (uint32_t)sum;
        } else {
          float sum = acc[0][nb][e];
#pragma unroll
          for (int c = 1; c < CH; ++c) sum += acc[c][nb][e];
          v[nb][e] = __float_as_uint(sum);
        }
      }
    const int z = zg / G, g = zg % G;
    if (!(chf == 0 && chl == C - 1)) {
      const long long ub = (long long)zg * C;
      const int f = cta_of(ub), l = cta_of(ub + C - 1);
      uint32_t* part = reinterpret_cast<uint32_t*>(a.partials);
      auto slot_base = [&](int c) -> uint32_t* {
        const long long cu0 = (long long)c * U / P;
        const int slot = (zg == (int)(cu0 / C)) ? 0 : 1;
        return part + ((size_t)(c * 2 + slot) * 128) * TOK;
      };
      uint32_t* mine = slot_base(cta);
#pragma unroll
      for (int nb = 0; nb < NB; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e)
          mine[(16 * w + pr + (e >> 1) * 8) * TOK + nb * 8 + 2 * t + (e & 1)] = v[nb][e];
      __threadfence();
      named_bar_sync(1, kConsumerWarps * 32);
      if (threadIdx.x == 0) {
        const unsigned int prev = atomicAdd(a.tile_counters + f, 1u);
        const int is_last = prev == (unsigned int)(l - f);
        if (is_last) a.tile_counters[f] = 0u;
        s_flag = is_last;
      }
      named_bar_sync(1, kConsumerWarps * 32);
      if (!s_flag) return;
      __threadfence();
      // Sum the contributors' partial tiles with RU loads in flight per value: accumulator j takes
      // contributors f + j, f + j + RU, ... in order, then the RU accumulators are added pairwise.
      // The order depends only on (f, l), so the fp32 result is the same on every run.
      constexpr int RU = NB >= 8 ? 1 : 8 / NB;
      uint32_t ra[RU][NB][4];
#pragma unroll
      for (int j = 0; j < RU; ++j)
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
#pragma unroll
          for (int e = 0; e < 4; ++e) ra[j][nb][e] = 0u;
      auto add = [](uint32_t x, uint32_t y) -> uint32_t {
        return kInt8 ? (uint32_t)((int)x + (int)y) : __float_as_uint(__uint_as_float(x) + __uint_as_float(y));
      };
      for (int c0 = f; c0 <= l; c0 += RU) {
#pragma unroll
        for (int j = 0; j < RU; ++j) {
          if (c0 + j > l) break;
          const uint32_t* src = slot_base(c0 + j);
#pragma unroll
          for (int nb = 0; nb < NB; ++nb)
#pragma unroll
            for (int e = 0; e < 4; ++e)
              ra[j][nb][e] = add(ra[j][nb][e],
                                 __ldcg(src + (16 * w + pr + (e >> 1) * 8) * TOK + nb * 8 + 2 * t + (e & 1)));
        }
      }
#pragma unroll
      for (int span = 1; span < RU; span <<= 1)
#pragma unroll
        for (int j = 0; j + span < RU; j += 2 * span)
#pragma unroll
          for (int nb = 0; nb < NB; ++nb)
#pragma unroll
            for (int e = 0; e < 4; ++e) ra[j][nb][e] = add(ra[j][nb][e], ra[j + span][nb][e]);
#pragma unroll
      for (int nb = 0; nb < NB; ++nb)
#pragma unroll
        for (int e = 0; e < 4; ++e) v[nb][e] = ra[0][nb][e];
    }
    epilogue(z, g, v);
  };

  zero_acc();
  int cur = -1, chf = 0, chl = 0;
  long long it = 0;
  const uint32_t rowA = (uint32_t)(16 * w + pr) * 128u, rowB = rowA + 8u * 128u;
  for (long long u = u0; u < u1; ++u, ++it) {
    const int zg = (int)(u / C), ch = (int)(u % C);
    if (zg != cur) {
      if (cur >= 0) flush(cur, chf, chl);
      cur = zg;
      chf = ch;
      zero_acc();
    }
    chl = ch;
    const int s = (int)(it % S);
    const uint32_t ph = (uint32_t)((it / S) & 1);
    if (ok) {
      bool got = true;
      if (lane == 0) got = mbar_wait_bounded(smem_u32(full + s), ph, kWaitBudgetCycles);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        ok = false;
        if (lane == 0) atomicOr(a.err, DEVERR_CONSUMER_WAIT);
      }
    }
    if (!ok) continue;  // no data: skip the math and do not release the stage

    const uint32_t sb = ring + (uint32_t)s * SB;
#pragma unroll
    for (int st = 0; st < STEPS; ++st) {
      uint4 wa[2], wb[2];
      if constexpr (kInt8) {
        // weight box st/2, logical 16-byte chunk 4(st%2) + t of rows pr and pr+8 (row & 7 == pr)
        const uint32_t wbox = sb + (uint32_t)(st >> 1) * kBox;
        const uint32_t off = (uint32_t)(((4 * (st & 1) + t) ^ pr) << 4);
        wa[0] = lds128(wbox + rowA + off);
        wb[0] = lds128(wbox + rowB + off);
      } else {
        // weight box st, logical chunks 2t and 2t+1 of rows gl and gl+8
        const uint32_t wbox = sb + (uint32_t)st * kBox;
        const uint32_t o0 = (uint32_t)(((2 * t) ^ pr) << 4), o1 = (uint32_t)(((2 * t + 1) ^ pr) << 4);
        wa[0] = lds128(wbox + rowA + o0);
        wa[1] = lds128(wbox + rowA + o1);
        wb[0] = lds128(wbox + rowB + o0);
        wb[1] = lds128(wbox + rowB + o1);
      }
      // A fragments of the four MMAs of this step (INT8 codes widened to fp16 in registers)
      uint32_t af[4][4];
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        if constexpr (kInt8) {
          i8x4_to_f16x2x2(u4c(wa[0], j), af[j][0], af[j][2]);
          i8x4_to_f16x2x2(u4c(wb[0], j), af[j][1], af[j][3]);
        } else {
          af[j][0] = u4c(wa[j >> 1], (2 * j) & 3);
          af[j][2] = u4c(wa[j >> 1], (2 * j + 1) & 3);
          af[j][1] = u4c(wb[j >> 1], (2 * j) & 3);
          af[j][3] = u4c(wb[j >> 1], (2 * j + 1) & 3);
        }
      }
      const uint32_t xbox = sb + 2 * kBox + (uint32_t)st * XBOX;
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const uint32_t xr = xbox + (uint32_t)(nb * 8 + gl) * 128u;  // token row & 7 == gl
        const uint4 x0 = lds128(xr + (uint32_t)(((2 * t) ^ gl) << 4));
        const uint4 x1 = lds128(xr + (uint32_t)(((2 * t + 1) ^ gl) << 4));
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const uint4& xv = (j >> 1) ? x1 : x0;
          const uint32_t b0 = u4c(xv, (2 * j) & 3);
          const uint32_t b1 = u4c(xv, (2 * j + 1) & 3);
          if constexpr (kInt8)
            mma_f16_16816(acc[j % CH][nb], af[j][0], af[j][1], af[j][2], af[j][3], b0, b1);
          else
            mma_bf16_16816(acc[j % CH][nb], af[j][0], af[j][1], af[j][2], af[j][3], b0, b1);
        }
      }
    }
    if constexpr (kInt8) {
      since += STEPS;
      if (since >= 16) {  // 16 steps = 1024 k: every partial sum so far is below 2^24
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
#pragma unroll
            for (int c = 0; c < CH; ++c) {
              iacc[nb][e] += __float2int_rn(acc[c][nb][e]);
              acc[c][nb][e] = 0.0f;
            }
          }
        since = 0;
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(empty + s));
  }
  if (cur >= 0) flush(cur, chf, chl);
  if (!want_top) return;
  // top-1 across the grid: every CTA publishes its maxima, then counts itself once; the last CTA
  // decodes the keys into indices and clears them
  publish_top();
  __threadfence();
  named_bar_sync(1, kConsumerWarps * 32);
  if (threadIdx.x == 0) {
    const unsigned int prev = atomicAdd(a.grid_counter, 1u);
    s_flag = prev == (unsigned int)(P - 1);
    if (s_flag) *a.grid_counter = 0u;
  }
  named_bar_sync(1, kConsumerWarps * 32);
  if (!s_flag) return;
  __threadfence();
  for (int tk = threadIdx.x; tk < a.M; tk += kConsumerWarps * 32) {
    const unsigned long long key = atomicExch(a.top_keys + tk, 0ull);
    a.top1[tk] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
  }
}

template <bool kInt8, int NB, int STEPS>
w8a8_status launch_steps(const StreamArgs& a, cudaStream_t st) {
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(stream_gemm_kernel<kInt8, NB, STEPS>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemLimit / Cps<NB>::value - kStaticReserve));
    attr_set[dev] = true;
  }
  constexpr int EB = kInt8 ? 1 : 2;
  CUtensorMap tw, tx;
  W8A8_TRY(make_tmap_2d(&tw, a.W, EB, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K * EB, 128 / EB, 128));
  W8A8_TRY(make_tmap_2d(&tx, a.X, 2, (uint64_t)a.K, (uint64_t)a.M, (uint64_t)a.K * 2, 64, 8 * NB));
  W8A8_CUDA(launch_pdl(stream_gemm_kernel<kInt8, NB, STEPS>, dim3(a.p.P), dim3(kThreads), a.p.smem_bytes, st, tw, tx,
                       a));
  return W8A8_OK;
}

template <bool kInt8, int NB>
w8a8_status launch_nb(const StreamArgs& a, cudaStream_t st) {
  constexpr int full = Geo<kInt8>::KCMAX / 64;
  return a.p.KC == Geo<kInt8>::KCMAX ? launch_steps<kInt8, NB, full>(a, st) : launch_steps<kInt8, NB, full / 2>(a, st);
}

template <bool kInt8>
w8a8_status launch_typed(const StreamArgs& a, cudaStream_t st) {
  switch (a.p.NB) {
    case 1: return launch_nb<kInt8, 1>(a, st);
    case 2: return launch_nb<kInt8, 2>(a, st);
    case 4: return launch_nb<kInt8, 4>(a, st);
    default: return launch_nb<kInt8, 8>(a, st);
  }
}

// ---------------------------------------------------------------------------------------------
// INT8 GEMV for M <= 4 tokens: dp4a on the INT8 codes of both operands (exact INT32 sums, no
// widening), the activation codes resident in shared memory for the whole kernel.  Same producer,
// unit decomposition, partial-tile protocol and epilogues as the MMA kernel.  Lane l of consumer
// warp w reads, in pass i, 16 bytes of tile row 16w + (l & 7) + 8 (i & 1) at logical chunk
// (l >> 3) + 4 (i >> 1): the 8 lanes of a shared-memory phase read one logical chunk of 8 rows
// whose swizzle keys differ, so the phase touches every bank once.
template <int MT, int NCH>
__global__ void __launch_bounds__(kThreads, 2)
    gemv_dp4a_kernel(const __grid_constant__ CUtensorMap tmW, const StreamArgs a) {
  constexpr int KC = NCH * 16;  // k bytes (= elements) per unit
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ int s_flag;
  __shared__ unsigned long long s_best[kConsumerWarps][MT];

  const StreamPlan& p = a.p;
  const int S = p.stages, SB = p.stage_bytes;
  const uint32_t raw_u32 = smem_u32(smem_raw);
  const uint32_t ring = (raw_u32 + 1023u) & ~1023u;
  const uint32_t xs = ring + (uint32_t)S * SB;                      // X codes [MT][K] (+ zero tail)
  const uint32_t xbytes = (uint32_t)((MT * a.K + KC + 15) / 16 * 16);
  uint64_t* full = reinterpret_cast<uint64_t*>(smem_raw + (ring - raw_u32) + (size_t)S * SB + xbytes);
  uint64_t* empty = full + S;

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int G = p.G, C = p.C;
  const long long U = (long long)G * C;
  const int P = gridDim.x, cta = blockIdx.x;
  const long long u0 = p.whole ? (long long)cta * G / P * C : (long long)cta * U / P;
  const long long u1 = p.whole ? (long long)(cta + 1) * G / P * C : (long long)(cta + 1) * U / P;
  auto cta_of = [&](long long u) -> int { return (int)(((u + 1) * P + U - 1) / U - 1); };

  pdl_trigger();
  if (threadIdx.x == kConsumerWarps * 32) {  // the producer thread: fetch the tensor map before the first copy needs it
    prefetch_tmap(&tmW);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(smem_u32(full + s), 1);
      mbar_init(smem_u32(empty + s), kConsumerWarps);
    }
    fence_mbar_init();
  }
  __syncthreads();
  if (u0 >= u1) {
    pdl_wait();
    return;
  }

  // The producer streams weights only (independent of the preceding kernel) and starts at once;
  // the consumers wait for the preceding kernel, then stage the activation codes.
  if (warp == kConsumerWarps) {  // ---------------------------------------------- producer thread
    if (lane != 0) return;
    constexpr int nw = KC / 128;
    bool ok = true;
    long long it = 0;
    const uint64_t wpol = l2_evict_first_policy();  // every weight box is read once per call
    for (long long u = u0; u < u1; ++u, ++it) {
      const int s = (int)(it % S);
      const uint32_t ph = (uint32_t)((it / S) & 1);
      if (!mbar_wait_bounded(smem_u32(empty + s), ph ^ 1u, kWaitBudgetCycles)) {
        ok = false;
        break;
      }
      const int g = (int)(u / C), ch = (int)(u % C);
      const uint32_t bar = smem_u32(full + s);
      mbar_arrive_expect_tx(bar, (uint32_t)(nw * kBox));
      for (int b = 0; b < nw; ++b)
        tma_load_2d_policy(ring + (uint32_t)s * SB + b * kBox, &tmW, ch * KC + b * 128, g * 128, bar, wpol);
    }
    if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
    for (long long j = it > S ? it - S : 0; j < it; ++j) {
      if (!mbar_wait_bounded(smem_u32(full + (int)(j % S)), (uint32_t)((j / S) & 1), kWaitBudgetCycles)) {
        atomicOr(a.err, DEVERR_DRAIN_WAIT);
        break;
      }
    }
    return;
  }

  // ------------------------------------------------------------------------ consumer warps
  pdl_wait();
  {  // activation codes -> shared memory (tokens >= M and the tail past K are zero)
    const int8_t* X = reinterpret_cast<const int8_t*>(a.X);
    uint8_t* xsp = smem_raw + (xs - raw_u32);
    for (uint32_t i = threadIdx.x; i < xbytes / 16; i += kConsumerWarps * 32) {
      const uint32_t byte = i * 16;
      const int m = (int)(byte / (uint32_t)a.K), k = (int)(byte % (uint32_t)a.K);
      uint4 v = make_uint4(0, 0, 0, 0);
      if (m < a.M) v = *reinterpret_cast<const uint4*>(X + (size_t)m * a.K + k);
      *reinterpret_cast<uint4*>(xsp + byte) = v;
    }
  }
  named_bar_sync(1, kConsumerWarps * 32);
  const int w = warp, rl = lane & 7, cq = lane >> 3;
  const bool want_top = a.kind == EPI_F32 && a.top1 != nullptr;
  int acc[2][MT];
  bool ok = true;
  if (want_top)
    for (int i = lane; i < MT; i += 32) s_best[w][i] = 0ull;
  __syncwarp();

  auto zero_acc = [&]() {
#pragma unroll
    for (int q = 0; q < 2; ++q)
#pragma unroll
      for (int m = 0; m < MT; ++m) acc[q][m] = 0;
  };

  auto epilogue = [&](int g, int (&v)[2][MT]) {  // lanes 0..7 hold rows 16w + rl and 16w + rl + 8
    const int ra = g * 128 + 16 * w + rl, rb = ra + 8;
#pragma unroll
    for (int m = 0; m < MT; ++m) {
      unsigned long long best = 0ull;
      if (lane < 8 && m < a.M) {
        if (a.kind == EPI_GEGLU) {
          if (rb < a.N) {
            float gv = __fmul_rn(__fmul_rn(a.s_x[m], a.s_w[ra]), __int2float_rn(v[0][m]));
            float uv = __fmul_rn(__fmul_rn(a.s_x[m], a.s_w[rb]), __int2float_rn(v[1][m]));
            if (a.bias) {
              gv = __fadd_rn(gv, a.bias[ra]);
              uv = __fadd_rn(uv, a.bias[rb]);
            }
            if (a.acc_dbg) {
              a.acc_dbg[(size_t)m * a.N + ra] = v[0][m];
              a.acc_dbg[(size_t)m * a.N + rb] = v[1][m];
            }
            a.y[(size_t)m * (a.N >> 1) + ((g * 128 + 16 * w) >> 1) + rl] = f32_to_bf16_bits(geglu_recipe(gv, uv));
          }
        } else {
#pragma unroll
          for (int side = 0; side < 2; ++side) {
            const int i = side ? rb : ra;
            if (i >= a.N) continue;
            float y = __fmul_rn(__fmul_rn(a.s_x[m], a.s_w[i]), __int2float_rn(v[side][m]));
            if (a.bias) y = __fadd_rn(y, a.bias[i]);
            if (a.acc_dbg) a.acc_dbg[(size_t)m * a.N + i] = v[side][m];
            if (a.kind == EPI_BF16) {
              a.y[(size_t)m * a.N + i] = f32_to_bf16_bits(y);
            } else {
              if (a.logits) a.logits[(size_t)m * a.N + i] = y;
              const unsigned long long key =
                  ((unsigned long long)float_order_key(y) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)i);
              best = key > best ? key : best;
            }
          }
        }
      }
      if (want_top) {
#pragma unroll
        for (int o = 1; o < 8; o <<= 1) {
          const unsigned long long other = __shfl_xor_sync(0xffffffffu, best, o);
          best = other > best ? other : best;
        }
        if (lane == 0 && best > s_best[w][m]) s_best[w][m] = best;
      }
    }
  };

  auto flush = [&](int g, int chf, int chl) {
    int v[2][MT];
#pragma unroll
    for (int q = 0; q < 2; ++q)
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        int x = acc[q][m];
        x += __shfl_xor_sync(0xffffffffu, x, 8);
        x += __shfl_xor_sync(0xffffffffu, x, 16);
        v[q][m] = x;
      }
    if (!(chf == 0 && chl == C - 1)) {
      const long long ub = (long long)g * C;
      const int f = cta_of(ub), l = cta_of(ub + C - 1);
      int* part = reinterpret_cast<int*>(a.partials);
      auto slot_base = [&](int c) -> int* {
        const long long cu0 = (long long)c * U / P;
        const int slot = (g == (int)(cu0 / C)) ? 0 : 1;
        return part + ((size_t)(c * 2 + slot) * 128) * MT;
      };
      if (lane < 8) {
        int* mine = slot_base(cta);
#pragma unroll
        for (int q = 0; q < 2; ++q)
#pragma unroll
          for (int m = 0; m < MT; ++m) mine[(16 * w + rl + 8 * q) * MT + m] = v[q][m];
      }
      __threadfence();
      named_bar_sync(1, kConsumerWarps * 32);
      if (threadIdx.x == 0) {
        const unsigned int prev = atomicAdd(a.tile_counters + f, 1u);
        const int is_last = prev == (unsigned int)(l - f);
        if (is_last) a.tile_counters[f] = 0u;
        s_flag = is_last;
      }
      named_bar_sync(1, kConsumerWarps * 32);
      if (!s_flag) return;
      __threadfence();
      // All 32 lanes sum: lane rl + 8 cq takes contributors f + cq, f + cq + 4, ..., four at a time
      // (16 loads in flight per lane), then the four lane groups are added (INT32: any order).
#pragma unroll
      for (int q = 0; q < 2; ++q)
#pragma unroll
        for (int m = 0; m < MT; ++m) v[q][m] = 0;
      for (int c0 = f + cq; c0 <= l; c0 += 16) {
        int x[4][2][MT];
#pragma unroll
        for (int j = 0; j < 4; ++j) {
          const int c = c0 + 4 * j;
#pragma unroll
          for (int q = 0; q < 2; ++q)
#pragma unroll
            for (int m = 0; m < MT; ++m) x[j][q][m] = c <= l ? __ldcg(slot_base(c) + (16 * w + rl + 8 * q) * MT + m) : 0;
        }
#pragma unroll
        for (int j = 0; j < 4; ++j)
#pragma unroll
          for (int q = 0; q < 2; ++q)
#pragma unroll
            for (int m = 0; m < MT; ++m) v[q][m] += x[j][q][m];
      }
#pragma unroll
      for (int q = 0; q < 2; ++q)
#pragma unroll
        for (int m = 0; m < MT; ++m) {
          v[q][m] += __shfl_xor_sync(0xffffffffu, v[q][m], 8);
          v[q][m] += __shfl_xor_sync(0xffffffffu, v[q][m], 16);
        }
    }
    epilogue(g, v);
  };

  zero_acc();
  int cur = -1, chf = 0, chl = 0;
  long long it = 0;
  for (long long u = u0; u < u1; ++u, ++it) {
    const int g = (int)(u / C), ch = (int)(u % C);
    if (g != cur) {
      if (cur >= 0) flush(cur, chf, chl);
      cur = g;
      chf = ch;
      zero_acc();
    }
    chl = ch;
    const int s = (int)(it % S);
    const uint32_t ph = (uint32_t)((it / S) & 1);
    if (ok) {
      bool got = true;
      if (lane == 0) got = mbar_wait_bounded(smem_u32(full + s), ph, kWaitBudgetCycles);
      got = __shfl_sync(0xffffffffu, got, 0);
      if (!got) {
        ok = false;
        if (lane == 0) atomicOr(a.err, DEVERR_CONSUMER_WAIT);
      }
    }
    if (!ok) continue;
    const uint32_t wbase = ring + (uint32_t)s * SB + (uint32_t)(16 * w + rl) * 128u;
    const uint32_t xk = xs + (uint32_t)(ch * KC);
#pragma unroll
    for (int i = 0; i < NCH / 2; ++i) {
      const int q = i & 1, c = cq + 4 * (i >> 1);
      const uint4 wv = lds128(wbase + (uint32_t)q * 8u * 128u + (uint32_t)(c >> 3) * kBox + (uint32_t)(((c & 7) ^ rl) << 4));
#pragma unroll
      for (int m = 0; m < MT; ++m) {
        const uint4 xv = lds128(xk + (uint32_t)(m * a.K + 16 * c));
        int r = acc[q][m];
        r = __dp4a((int)wv.x, (int)xv.x, r);
        r = __dp4a((int)wv.y, (int)xv.y, r);
        r = __dp4a((int)wv.z, (int)xv.z, r);
        r = __dp4a((int)wv.w, (int)xv.w, r);
        acc[q][m] = r;
      }
    }
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_u32(empty + s));
  }
  if (cur >= 0) flush(cur, chf, chl);
  if (!want_top) return;
  __syncwarp();
  if (lane < MT && lane < a.M && s_best[w][lane] != 0ull) atomicMax(a.top_keys + lane, s_best[w][lane]);
  __threadfence();
  named_bar_sync(1, kConsumerWarps * 32);
  if (threadIdx.x == 0) {
    const unsigned int prev = atomicAdd(a.grid_counter, 1u);
    s_flag = prev == (unsigned int)(P - 1);
    if (s_flag) *a.grid_counter = 0u;
  }
  named_bar_sync(1, kConsumerWarps * 32);
  if (!s_flag) return;
  __threadfence();
  for (int tk = threadIdx.x; tk < a.M; tk += kConsumerWarps * 32) {
    const unsigned long long key = atomicExch(a.top_keys + tk, 0ull);
    a.top1[tk] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
  }
}

template <int MT, int NCH>
w8a8_status launch_dp4a(const StreamArgs& a, cudaStream_t st) {
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(gemv_dp4a_kernel<MT, NCH>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   kSmemLimit / 2 - kStaticReserve));
    attr_set[dev] = true;
  }
  CUtensorMap tw;
  W8A8_TRY(make_tmap_2d(&tw, a.W, 1, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K, 128, 128));
  W8A8_CUDA(launch_pdl(gemv_dp4a_kernel<MT, NCH>, dim3(a.p.P), dim3(kThreads), a.p.smem_bytes, st, tw, a));
  return W8A8_OK;
}

template <int MT>
w8a8_status launch_dp4a_mt(const StreamArgs& a, cudaStream_t st) {
  return a.p.KC == 256 ? launch_dp4a<MT, 16>(a, st) : launch_dp4a<MT, 8>(a, st);
}

}  // namespace

StreamPlan make_stream_plan(bool int8_weights, int M, int N, int K, int sm_count) {
  StreamPlan p{};
  if (int8_weights && M <= 4 && (size_t)4 * K <= 32768) {
    // INT8 GEMV with dp4a: X codes resident, two CTAs per SM, a stage = up to 2 weight boxes
    p.dp4a = 1;
    p.MT = M <= 1 ? 1 : M <= 2 ? 2 : 4;
    p.NB = 1;
    p.TOK = p.MT;
    p.Z = 1;
    p.G = std::max(1, (N + 127) / 128);
    p.KC = 256;
    while (p.KC > 128 && (long long)p.G * ((K + p.KC - 1) / p.KC) < 2 * sm_count) p.KC >>= 1;
    p.C = std::max(1, (K + p.KC - 1) / p.KC);
    p.P = (int)std::max(1LL, std::min<long long>(std::min(2 * sm_count, kTileCounterSlots), (long long)p.G * p.C));
    p.whole = p.G >= p.P;
    if (p.whole) p.KC = 256, p.C = std::max(1, (K + 255) / 256);
    p.stage_bytes = 2 * kBox;
    const int xbytes = (p.MT * K + p.KC + 15) / 16 * 16;
    p.stages = std::max(2, std::min(8, (kSmemLimit / 2 - kStaticReserve - 2048 - xbytes) / p.stage_bytes));
    p.smem_bytes = p.stages * p.stage_bytes + xbytes + 16 * p.stages + 1024;
    p.partial_bytes = (size_t)p.P * 2 * 128 * p.MT * 4;
    return p;
  }
  p.NB = M <= 8 ? 1 : M <= 16 ? 2 : M <= 32 ? 4 : 8;
  p.TOK = 8 * p.NB;
  p.Z = std::max(1, (M + p.TOK - 1) / p.TOK);
  p.G = std::max(1, (N + 127) / 128);
  // Largest chunk (256, 128 or 64 k elements; the stage holds up to Geo::KC) that still gives every
  // SM a unit; the grid never exceeds the number of units, so every CTA contributes.
  const int kcmax = int8_weights ? Geo<true>::KCMAX : Geo<false>::KCMAX;
  const int kcmin = int8_weights ? 128 : 64;  // one weight box
  p.KC = kcmax;
  while (p.KC > kcmin && (long long)p.Z * p.G * ((K + p.KC - 1) / p.KC) < sm_count) p.KC >>= 1;
  p.C = std::max(1, (K + p.KC - 1) / p.KC);
  const long long units = (long long)p.Z * p.G * p.C;
  const int cps = p.NB <= 4 ? 2 : 1;  // CTAs per SM (matches Cps<NB>)
  p.P = (int)std::max(1LL, std::min<long long>(std::min(cps * sm_count, kTileCounterSlots), units));
  p.whole = (long long)p.Z * p.G >= p.P;
  if (p.whole) {
    p.KC = kcmax;
    p.C = std::max(1, (K + p.KC - 1) / p.KC);
  }
  p.stage_bytes = stage_bytes_for(int8_weights, p.TOK);
  p.stages = std::max(2, std::min(8, (kSmemLimit / cps - kStaticReserve - 2048) / p.stage_bytes));
  p.smem_bytes = p.stages * p.stage_bytes + 16 * p.stages + 1024;  // + alignment slack for the ring
  p.partial_bytes = (size_t)p.P * 2 * 128 * p.TOK * 4;
  return p;
}

static thread_local cudaEvent_t g_ev_start = nullptr, g_ev_stop = nullptr;

void set_kernel_events(void* start, void* stop) {
  g_ev_start = reinterpret_cast<cudaEvent_t>(start);
  g_ev_stop = reinterpret_cast<cudaEvent_t>(stop);
}

void take_kernel_events(void** start, void** stop) {
  *start = g_ev_start;
  *stop = g_ev_stop;
  g_ev_start = g_ev_stop = nullptr;
}

static w8a8_status dispatch_stream_gemm(bool int8_weights, const StreamArgs& a, cudaStream_t st);

w8a8_status launch_stream_gemm(bool int8_weights, const StreamArgs& a, cudaStream_t st) {
  if (a.M == 0 || a.N == 0) return W8A8_OK;
  void *v0, *v1;
  take_kernel_events(&v0, &v1);
  cudaEvent_t e0 = reinterpret_cast<cudaEvent_t>(v0), e1 = reinterpret_cast<cudaEvent_t>(v1);
  if (e0) W8A8_CUDA(cudaEventRecord(e0, st));
  const w8a8_status s = dispatch_stream_gemm(int8_weights, a, st);
  if (e1) W8A8_CUDA(cudaEventRecord(e1, st));
  return s;
}

static w8a8_status dispatch_stream_gemm(bool int8_weights, const StreamArgs& a, cudaStream_t st) {
  W8A8_CHECK_ARG(!(a.kind == EPI_F32 && a.top1) || a.M <= kMaxTopKeys, W8A8_ERR_SHAPE,
                 "top-1: M=%d exceeds %d tokens per call", a.M, kMaxTopKeys);
  W8A8_CHECK_ARG(a.p.smem_bytes <= kSmemLimit / (a.p.NB == 1 ? 2 : 1) - kStaticReserve, W8A8_ERR_SHAPE,
                 "stream GEMM: stage does not fit in shared memory");
  if (a.p.dp4a) {
    W8A8_CHECK_ARG(int8_weights, W8A8_ERR_INVALID_ARG, "dp4a plan for bf16 weights");
    switch (a.p.MT) {
      case 1: return launch_dp4a_mt<1>(a, st);
      case 2: return launch_dp4a_mt<2>(a, st);
      default: return launch_dp4a_mt<4>(a, st);
    }
  }
  return int8_weights ? launch_typed<true>(a, st) : launch_typed<false>(a, st);
}

void attach_reserved(StreamArgs& a, void* ws) {
  char* base = reinterpret_cast<char*>(ws);
  a.tile_counters = reinterpret_cast<unsigned int*>(base);
  a.grid_counter = reinterpret_cast<unsigned int*>(base + kGridCounterOffset);
  a.top_keys = reinterpret_cast<unsigned long long*>(base + kTopKeysOffset);
  a.err = reinterpret_cast<unsigned int*>(base + kErrWordOffset);
}

int max_top_keys() { return kMaxTopKeys; }

}  // namespace w8a8
