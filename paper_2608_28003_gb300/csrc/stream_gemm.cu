// Weight-streaming GEMM for decode-sized token counts, legacy tensor-core MMA (m16n8k16).
//
// Computes acc_ti = sum_j X_tj * W_ij for W [N, K] (row = output channel) and X [M, K]
// (Eq. gemm-final for the W8A8 path; the bf16 pass-through of the FFN section otherwise), then
// the epilogue of the calling layer.  The weights are the streamed operand (decode is
// HBM-bound on them); tokens ride in the MMA's N dimension (8 per block).
//
// W8A8 path: INT8 codes are loaded straight from global memory into registers and widened to
// fp16 in registers (exact); X arrives as fp16 codes.  fp16 x fp16 products of codes are exact
// integers below 2^14 and every partial sum of at most 1024 products stays below 2^24, where
// fp32 represents integers exactly, so each warp folds its fp32 accumulator into INT32 every
// 16 k-steps (1024 k): the INT32 result is exact whatever order the hardware adds in.
//
// Fragment layout: lane = 4g + t.  In a 64-wide k step the lane loads k = 16t .. 16t+15 of
// weight rows g and g+8 and of token g.  The m16n8k16 fragments of MMA j (j = 0..3) take the
// lane's k = 16t+4j .. 16t+4j+3 for both operands, so every MMA pairs the same physical k on
// A and B, and the four MMAs of a step cover all 64 k: a k permutation that a dot product
// does not see.
//
// Work split: 16-row tiles x k slices; a CTA holds RPC row tiles x WS k slices (one warp
// each) and reduces its slices in shared memory.  Small-N layers also split k across CTAs
// (CS > 1): each CTA writes its partial tile, and the last CTA to arrive (an atomic counter,
// no waiting) sums the partials in a fixed order and runs the epilogue.  INT32 partials make
// this exact; fp32 partials (bf16 path) are summed in a fixed order, so results are
// deterministic.
#include <algorithm>

#include "stream_gemm.cuh"

namespace w8a8 {

namespace {

__device__ __forceinline__ uint32_t u4c(const uint4& v, int c) {
  return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

constexpr int kTileCounterSlots = 8192;                    // uint32 slots at workspace offset 0
constexpr size_t kGridCounterOffset = 8192 * 4;            // one uint32
constexpr size_t kTopKeysOffset = 40960;                   // uint64 keys
constexpr int kMaxTopKeys = (W8A8_WS_RESERVED - 40960) / 8;  // 3072

template <bool kInt8, int NB, int U>
__global__ void __launch_bounds__(256) stream_gemm_kernel(const StreamArgs a) {
  constexpr int TOK = 8 * NB;
  constexpr int WV = kInt8 ? 1 : 2;  // 16-byte vectors per 16-k weight chunk
  constexpr int EB = kInt8 ? 1 : 2;  // weight element bytes
  __shared__ uint32_t red[8 * 16 * TOK];
  __shared__ unsigned long long skeys[TOK];
  __shared__ int s_last;

  const StreamPlan& p = a.p;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int g = lane >> 2, t = lane & 3;
  const int group = blockIdx.x / p.CS, cs = blockIdx.x % p.CS;
  const int z = blockIdx.z;
  const int tok0 = z * TOK;
  const int rt_local = warp / p.WS, ws = warp % p.WS;
  const int rt = group * p.RPC + rt_local;
  const int sl = cs * p.WS + ws;
  const int s_begin = sl * p.sps;
  const int s_end = rt < p.RT ? min(p.KS, s_begin + p.sps) : s_begin;
  const bool want_top = a.kind == EPI_F32 && a.top1 != nullptr;

  if (want_top)
    for (int i = threadIdx.x; i < TOK; i += blockDim.x) skeys[i] = 0ull;

  const int row_a = rt * 16 + g, row_b = row_a + 8;
  const bool va = row_a < a.N, vb = row_b < a.N;
  const char* wa_ptr = reinterpret_cast<const char*>(a.W) + (size_t)(va ? row_a : 0) * a.K * EB;
  const char* wb_ptr = reinterpret_cast<const char*>(a.W) + (size_t)(vb ? row_b : 0) * a.K * EB;

  float acc[NB][4];
  int iacc[NB][4];
#pragma unroll
  for (int nb = 0; nb < NB; ++nb)
#pragma unroll
    for (int e = 0; e < 4; ++e) {
      acc[nb][e] = 0.0f;
      iacc[nb][e] = 0;
    }
  int since = 0;
  const uint4 zero4 = make_uint4(0, 0, 0, 0);

  for (int s0 = s_begin; s0 < s_end; s0 += U) {
    uint4 wa[U][WV], wb[U][WV];
    uint4 xv[U][NB][2];
#pragma unroll
    for (int u = 0; u < U; ++u) {
      const int s = s0 + u;
      const int k = s * 64 + t * 16;
      const bool kv = (s < s_end) && (k < a.K);
#pragma unroll
      for (int v = 0; v < WV; ++v) {
        wa[u][v] = (kv && va) ? ldg_stream(wa_ptr + (size_t)k * EB + 16 * v) : zero4;
        wb[u][v] = (kv && vb) ? ldg_stream(wb_ptr + (size_t)k * EB + 16 * v) : zero4;
      }
#pragma unroll
      for (int nb = 0; nb < NB; ++nb) {
        const int tok = tok0 + nb * 8 + g;
        const bool tv = kv && tok < a.M;
        const uint16_t* xp = a.X + (size_t)(tv ? tok : 0) * a.K + (tv ? k : 0);
        xv[u][nb][0] = tv ? ldg_keep(xp) : zero4;
        xv[u][nb][1] = tv ? ldg_keep(xp + 8) : zero4;
      }
    }
#pragma unroll
    for (int u = 0; u < U; ++u) {
#pragma unroll
      for (int j = 0; j < 4; ++j) {
        uint32_t a0, a1, a2, a3;
        if constexpr (kInt8) {
          i8x4_to_f16x2x2(u4c(wa[u][0], j), a0, a2);
          i8x4_to_f16x2x2(u4c(wb[u][0], j), a1, a3);
        } else {
          a0 = u4c(wa[u][j >> 1], (2 * j) & 3);
          a2 = u4c(wa[u][j >> 1], (2 * j + 1) & 3);
          a1 = u4c(wb[u][j >> 1], (2 * j) & 3);
          a3 = u4c(wb[u][j >> 1], (2 * j + 1) & 3);
        }
#pragma unroll
        for (int nb = 0; nb < NB; ++nb) {
          const uint32_t b0 = u4c(xv[u][nb][j >> 1], (2 * j) & 3);
          const uint32_t b1 = u4c(xv[u][nb][j >> 1], (2 * j + 1) & 3);
          if constexpr (kInt8)
            mma_f16_16816(acc[nb], a0, a1, a2, a3, b0, b1);
          else
            mma_bf16_16816(acc[nb], a0, a1, a2, a3, b0, b1);
        }
      }
    }
    if constexpr (kInt8) {
      since += U;
      if (since >= 16) {  // 16 steps = 1024 k: every partial sum so far is below 2^24
#pragma unroll
        for (int nb = 0; nb < NB; ++nb)
#pragma unroll
          for (int e = 0; e < 4; ++e) {
            iacc[nb][e] += __float2int_rn(acc[nb][e]);
            acc[nb][e] = 0.0f;
          }
        since = 0;
      }
    }
  }

  // ---- per-warp tile -> shared memory: red[warp][row][tok]
  {
    uint32_t* r = red + warp * 16 * TOK;
#pragma unroll
    for (int nb = 0; nb < NB; ++nb) {
      const int c0 = nb * 8 + 2 * t;
      uint32_t v[4];
#pragma unroll
      for (int e = 0; e < 4; ++e)
        v[e] = kInt8 ? (uint32_t)(iacc[nb][e] + __float2int_rn(acc[nb][e])) : __float_as_uint(acc[nb][e]);
      r[g * TOK + c0] = v[0];
      r[g * TOK + c0 + 1] = v[1];
      r[(g + 8) * TOK + c0] = v[2];
      r[(g + 8) * TOK + c0 + 1] = v[3];
    }
  }
  __syncthreads();

  // ---- reduce the WS slices of each row tile in place into slot ws = 0
  const int nthreads = blockDim.x;
  const int E = p.RPC * 16 * TOK;
  auto fin_index = [&](int e) {  // element e = (rtl * 16 + row) * TOK + tok
    const int rtl = e / (16 * TOK);
    const int rem = e - rtl * 16 * TOK;
    return (rtl * p.WS) * 16 * TOK + rem;
  };
  for (int e = threadIdx.x; e < E; e += nthreads) {
    const int rtl = e / (16 * TOK);
    const int rem = e - rtl * 16 * TOK;
    const uint32_t* base = red + (rtl * p.WS) * 16 * TOK + rem;
    if constexpr (kInt8) {
      int s = 0;
      for (int w = 0; w < p.WS; ++w) s += (int)base[w * 16 * TOK];
      red[fin_index(e)] = (uint32_t)s;
    } else {
      float s = 0.0f;
      for (int w = 0; w < p.WS; ++w) s += __uint_as_float(base[w * 16 * TOK]);
      red[fin_index(e)] = __float_as_uint(s);
    }
  }

  // ---- cross-CTA k split: partials + last-arriver reduction (no waiting)
  if (p.CS > 1) {
    uint32_t* part = reinterpret_cast<uint32_t*>(a.partials);
    const size_t rows_total = (size_t)p.RT * 16;
    for (int e = threadIdx.x; e < E; e += nthreads) {
      const int rtl = e / (16 * TOK);
      const int rem = e - rtl * 16 * TOK;
      const int rtg = group * p.RPC + rtl;
      if (rtg < p.RT) part[((size_t)(z * p.CS + cs) * rows_total + (size_t)rtg * 16) * TOK + rem] = red[fin_index(e)];
    }
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      unsigned int* ctr = a.tile_counters + z * p.groups + group;
      const unsigned int prev = atomicAdd(ctr, 1u);
      s_last = (prev == (unsigned int)(p.CS - 1));
      if (s_last) *ctr = 0u;  // every CTA of this tile has arrived: reset for the next call
    }
    __syncthreads();
    if (!s_last) return;
    __threadfence();
    for (int e = threadIdx.x; e < E; e += nthreads) {
      const int rtl = e / (16 * TOK);
      const int rem = e - rtl * 16 * TOK;
      const int rtg = group * p.RPC + rtl;
      if (rtg >= p.RT) continue;
      if constexpr (kInt8) {
        int s = 0;
        for (int c = 0; c < p.CS; ++c)
          s += (int)__ldcg(part + ((size_t)(z * p.CS + c) * rows_total + (size_t)rtg * 16) * TOK + rem);
        red[fin_index(e)] = (uint32_t)s;
      } else {
        float s = 0.0f;
        for (int c = 0; c < p.CS; ++c)
          s += __uint_as_float(__ldcg(part + ((size_t)(z * p.CS + c) * rows_total + (size_t)rtg * 16) * TOK + rem));
        red[fin_index(e)] = __float_as_uint(s);
      }
    }
  }
  __syncthreads();

  // ---- epilogue
  auto value_f32 = [&](int e, int i, int tk) -> float {  // dequantised fp32 value (before bias)
    const uint32_t r = red[fin_index(e)];
    if constexpr (kInt8) {
      const float sc = __fmul_rn(a.s_x[tk], a.s_w[i]);  // s_t^x * s_i^W
      return __fmul_rn(sc, __int2float_rn((int)r));
    } else {
      return __uint_as_float(r);
    }
  };
  if (a.kind == EPI_GEGLU) {
    const int E2 = p.RPC * 8 * TOK;
    const int F = a.N >> 1;
    for (int e2 = threadIdx.x; e2 < E2; e2 += nthreads) {
      const int rtl = e2 / (8 * TOK);
      const int rem = e2 - rtl * 8 * TOK;
      const int r = rem / TOK, tok = rem - (rem / TOK) * TOK;
      const int rtg = group * p.RPC + rtl;
      const int tk = tok0 + tok;
      const int ig = rtg * 16 + r, iu = ig + 8;
      if (rtg >= p.RT || iu >= a.N || tk >= a.M) continue;
      const int eg = (rtl * 16 + r) * TOK + tok, eu = (rtl * 16 + r + 8) * TOK + tok;
      float gv = value_f32(eg, ig, tk), uv = value_f32(eu, iu, tk);
      if (a.bias) {
        gv = __fadd_rn(gv, a.bias[ig]);
        uv = __fadd_rn(uv, a.bias[iu]);
      }
      if constexpr (kInt8) {
        if (a.acc_dbg) {
          a.acc_dbg[(size_t)tk * a.N + ig] = (int)red[fin_index(eg)];
          a.acc_dbg[(size_t)tk * a.N + iu] = (int)red[fin_index(eu)];
        }
      }
      a.y[(size_t)tk * F + rtg * 8 + r] = f32_to_bf16_bits(geglu_recipe(gv, uv));
    }
  } else {
    for (int e = threadIdx.x; e < E; e += nthreads) {
      const int rtl = e / (16 * TOK);
      const int rem = e - rtl * 16 * TOK;
      const int row = rem / TOK, tok = rem - row * TOK;
      const int rtg = group * p.RPC + rtl;
      const int i = rtg * 16 + row, tk = tok0 + tok;
      if (rtg >= p.RT || i >= a.N || tk >= a.M) continue;
      float y = value_f32(e, i, tk);
      if (a.bias) y = __fadd_rn(y, a.bias[i]);
      if constexpr (kInt8) {
        if (a.acc_dbg) a.acc_dbg[(size_t)tk * a.N + i] = (int)red[fin_index(e)];
      }
      if (a.kind == EPI_BF16) {
        a.y[(size_t)tk * a.N + i] = f32_to_bf16_bits(y);
      } else {
        if (a.logits) a.logits[(size_t)tk * a.N + i] = y;
        if (want_top) {
          const unsigned long long key =
              ((unsigned long long)float_order_key(y) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)i);
          atomicMax(&skeys[tok], key);
        }
      }
    }
  }

  // ---- top-1 across the grid: CTA maxima -> global keys; the last finalising CTA decodes them
  if (want_top) {
    __syncthreads();
    for (int i = threadIdx.x; i < TOK; i += blockDim.x)
      if (tok0 + i < a.M && skeys[i] != 0ull) atomicMax(a.top_keys + tok0 + i, skeys[i]);
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) {
      const unsigned int total = (unsigned int)(p.groups * p.zgroups);
      const unsigned int prev = atomicAdd(a.grid_counter, 1u);
      s_last = (prev == total - 1);
      if (s_last) *a.grid_counter = 0u;
    }
    __syncthreads();
    if (s_last) {
      __threadfence();
      for (int tk = threadIdx.x; tk < a.M; tk += nthreads) {
        const unsigned long long key = atomicExch(a.top_keys + tk, 0ull);
        a.top1[tk] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
      }
    }
  }
}

template <bool kInt8, int NB, int U>
w8a8_status launch_nb(const StreamArgs& a, cudaStream_t st) {
  const StreamPlan& p = a.p;
  dim3 grid(p.groups * p.CS, 1, p.zgroups);
  dim3 block(32 * p.RPC * p.WS);
  stream_gemm_kernel<kInt8, NB, U><<<grid, block, 0, st>>>(a);
  W8A8_LAUNCH_CHECK();
  return W8A8_OK;
}

template <bool kInt8>
w8a8_status launch_typed(const StreamArgs& a, cudaStream_t st) {
  switch (a.p.NB) {
    case 1: return launch_nb<kInt8, 1, 4>(a, st);
    case 2: return launch_nb<kInt8, 2, 4>(a, st);
    case 4: return launch_nb<kInt8, 4, 2>(a, st);
    default: return launch_nb<kInt8, 8, 1>(a, st);
  }
}

}  // namespace

StreamPlan make_stream_plan(int M, int N, int K, int sm_count) {
  StreamPlan p{};
  p.NB = M <= 8 ? 1 : M <= 16 ? 2 : M <= 32 ? 4 : 8;
  const int TOK = 8 * p.NB;
  p.zgroups = M > 0 ? (M + TOK - 1) / TOK : 1;
  p.RT = (N + 15) / 16;
  p.KS = std::max(1, (K + 63) / 64);
  const long target = std::max(1L, (long)sm_count * 16 / p.zgroups);
  long S = (target + p.RT - 1) / std::max(1, p.RT);
  S = std::max(1L, std::min((long)p.KS, S));
  p.sps = (p.KS + (int)S - 1) / (int)S;
  p.S = (p.KS + p.sps - 1) / p.sps;
  p.WS = std::min(p.S, 8);
  p.CS = (p.S + p.WS - 1) / p.WS;
  p.RPC = std::max(1, std::min(8 / p.WS, p.RT));
  p.groups = (p.RT + p.RPC - 1) / p.RPC;
  p.partial_bytes = p.CS > 1 ? (size_t)p.zgroups * p.CS * p.RT * 16 * TOK * 4 : 0;
  return p;
}

w8a8_status launch_stream_gemm(bool int8_weights, const StreamArgs& a, cudaStream_t st) {
  if (a.M == 0 || a.N == 0) return W8A8_OK;
  const StreamPlan& p = a.p;
  W8A8_CHECK_ARG(p.CS == 1 || p.zgroups * p.groups <= kTileCounterSlots, W8A8_ERR_SHAPE,
                 "stream GEMM: %d split tiles exceed the %d counter slots", p.zgroups * p.groups, kTileCounterSlots);
  W8A8_CHECK_ARG(!(a.kind == EPI_F32 && a.top1) || a.M <= kMaxTopKeys, W8A8_ERR_SHAPE,
                 "top-1: M=%d exceeds %d tokens per call", a.M, kMaxTopKeys);
  return int8_weights ? launch_typed<true>(a, st) : launch_typed<false>(a, st);
}

// Workspace carve-up shared by the entry points.
void attach_reserved(StreamArgs& a, void* ws) {
  char* base = reinterpret_cast<char*>(ws);
  a.tile_counters = reinterpret_cast<unsigned int*>(base);
  a.grid_counter = reinterpret_cast<unsigned int*>(base + kGridCounterOffset);
  a.top_keys = reinterpret_cast<unsigned long long*>(base + kTopKeysOffset);
}

int max_top_keys() { return kMaxTopKeys; }

}  // namespace w8a8
