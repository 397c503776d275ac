// Tensor-core GEMM (tcgen05, TMEM accumulators, TMA) for prefill-sized token counts.
//
// A persistent grid (one CTA per SM) walks the output tiles of 128 tokens x BN channels.  A
// (tokens x K) and B (channels x K) tiles of 64 k arrive by 2-D TMA into 128-byte-swizzled shared
// memory, S stages deep, continuously across tiles.  Accumulators live in tensor memory (all 512
// columns), as a ring of BN-column slots, so the epilogue of one tile overlaps the MMAs of the next.
//  * warp 4 (one thread) issues the TMA copies; warp 5 allocates tensor memory and one of its
//    threads issues tcgen05.mma (M = 128, N = BN, K = 16, fp32 accumulation) for each stage,
//    commits the stage back to the producer and each finished slot to the epilogue; warps 0-3 are
//    the epilogue, warp w reading TMEM lanes 32w .. 32w+31 (its tokens) with tcgen05.ld and
//    handing the slot back.
//  * W8A8 path (BN = 128, four slots): both operands are INT8 codes stored as fp16 (exact).  Every
//    product is an integer below 2^14, so a fp32 sum of at most 1024 of them is exact; the
//    accumulator is therefore restarted every 1024 k (16 stages) in the next slot while the
//    epilogue folds the finished one into INT32 registers, and the INT32 result is exact in any
//    order (Eq. gemm-final).  The epilogue then dequantises fl(fl(s_x s_w) acc) (+ bias).
//  * bf16 path (BN = 256 and two slots, or BN = 128 and four when 256-wide tiles would leave SMs
//    idle): one accumulator per tile over the whole k range.
//  * epilogues: bf16 output, GeGLU of interleaved gate/up columns (16-column blocks: 8 gate, then
//    the 8 matching up channels), or fp32 logits with the top-1 index (keys reduced with atomicMax,
//    the last CTA to finish decodes them).
// Every mbarrier wait is bounded: on timeout the kernel sets a bit of the error word, stops, waits
// (bounded) for its own copies and MMAs in flight and frees its tensor memory.
#include <algorithm>

#include "gemm_tc.cuh"
#include "ops.cuh"
#include "stream_gemm.cuh"
#include "tmap.cuh"

namespace w8a8 {

namespace {

constexpr int kBM = 128;
constexpr int kSwz = 128;                // swizzle span in bytes (TMA and the MMA descriptors agree)
constexpr int kBK = kSwz / 2;            // k per stage: one swizzle span of fp16 per row
constexpr int kKbPerChunk = 1024 / kBK;  // stages per exact fp32 chunk of 1024 k
constexpr int kThreads = 192;
constexpr uint32_t kTmemCols = 512;  // all of an SM's tensor memory: 2 (bf16) or 4 (W8A8) accumulator slots
constexpr uint32_t kABytes = kBM * kBK * 2;

template <bool kInt8, int kBN>
struct TcGeo {
  static constexpr int BN = kBN;
  static constexpr uint32_t BBytes = BN * kBK * 2;
  static constexpr int S = (192 * 1024) / (int)(kABytes + BBytes);
  static constexpr int Smem = S * (kABytes + BBytes) + 1024;
};

// ---------------------------------------------------------------------------- tcgen05 helpers
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major tile swizzled over kSwz bytes: rows of kSwz bytes,
// 8-row groups 8 kSwz bytes apart (stride byte offset), descriptor version 1, layout SWIZZLE_128B
// (2) or SWIZZLE_64B (4).
__device__ __forceinline__ uint64_t sdesc_swz(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                       // leading byte offset (unused by swizzled K-major layouts)
  d |= (uint64_t)((8 * kSwz) >> 4) << 32;       // stride byte offset
  d |= (uint64_t)1 << 46;                       // version
  d |= (uint64_t)(kSwz == 128 ? 2 : 4) << 61;   // layout
  return d;
}

// Instruction descriptor of kind::f16: fp32 accumulator, A/B fp16 (0) or bf16 (1), both K-major,
// N >> 3 at bit 17, M >> 4 at bit 24.
__host__ __device__ constexpr uint32_t idesc_f16(uint32_t ab_format, int n, int m) {
  return (1u << 4) | (ab_format << 7) | (ab_format << 10) | ((uint32_t)(n >> 3) << 17) | ((uint32_t)(m >> 4) << 24);
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                       uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr));
  asm volatile("tcgen05.wait::ld.sync.aligned;\n" ::: "memory");
}

__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  return (uint32_t)f32_to_bf16_bits(a) | ((uint32_t)f32_to_bf16_bits(b) << 16);
}

template <bool kInt8, int kBN>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB, const TcArgs a) {
  using GG = TcGeo<kInt8, kBN>;
  constexpr int BN = GG::BN, S = GG::S;
  constexpr int NSLOT = (int)kTmemCols / BN;  // accumulator slots in tensor memory
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t bars[2 * S + 2 * NSLOT + 1];
  __shared__ uint32_t tmem_slot;
  __shared__ int s_flag;

  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t sA = base, sB = base + (uint32_t)S * kABytes;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int NT = (a.N + BN - 1) / BN, tiles = NT * ((a.M + kBM - 1) / kBM);
  const int nkb = (a.K + kBK - 1) / kBK;
  const int nchunks = kInt8 ? (nkb + kKbPerChunk - 1) / kKbPerChunk : 1;
  const int kb_per_chunk = kInt8 ? kKbPerChunk : nkb;
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, accf0 = full0 + 16 * S, acce0 = accf0 + 8 * NSLOT,
                 done = acce0 + 8 * NSLOT;

  pdl_trigger();
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < NSLOT; ++b) {
      mbar_init(accf0 + 8 * b, 1);
      mbar_init(acce0 + 8 * b, 128);
    }
    mbar_init(done, 1);
    fence_mbar_init();
  }
  if (warp == 5) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(&tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;\n" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  pdl_wait();  // activations and outputs belong to the preceding kernels

  // Persistent: CTA b takes tiles b, b + grid, ...; tile t covers channels (t mod NT) * BN and
  // tokens (t / NT) * 128, so neighbouring CTAs share the activation rows.
  if (warp == 4) {
    // ---------------------------------------------------------------------- TMA producer
    if (lane == 0) {
      bool ok = true;
      int g = 0;  // stages issued
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        const int n0 = (t % NT) * BN, m0 = (t / NT) * kBM;
        for (int kb = 0; kb < nkb; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait_bounded(empty0 + 8 * s, (uint32_t)(((g / S) & 1) ^ 1), kWaitBudgetCycles)) {
            ok = false;
            break;
          }
          const uint32_t bar = full0 + 8 * s;
          mbar_arrive_expect_tx(bar, kABytes + GG::BBytes);
          tma_load_2d(sA + (uint32_t)s * kABytes, &tmA, kb * kBK, m0, bar);
          tma_load_2d(sB + (uint32_t)s * GG::BBytes, &tmB, kb * kBK, n0, bar);
        }
      }
      if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
      for (int j = g > S ? g - S : 0; j < g; ++j) {  // let the last copies land before exit
        if (!mbar_wait_bounded(full0 + 8 * (j % S), (uint32_t)((j / S) & 1), kWaitBudgetCycles)) {
          atomicOr(a.err, DEVERR_DRAIN_WAIT);
          break;
        }
      }
    }
  } else if (warp == 5) {
    // ---------------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16(kInt8 ? 0u : 1u, BN, kBM);
      bool ok = true;
      int g = 0, q = 0;  // stages consumed, accumulator chunks produced
      for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
        for (int c = 0; c < nchunks && ok; ++c, ++q) {
          const int slot = q % NSLOT;
          if (q >= NSLOT &&  // the epilogue has drained this slot's previous chunk
              !mbar_wait_bounded(acce0 + 8 * slot, (uint32_t)(((q / NSLOT) - 1) & 1), kWaitBudgetCycles)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint32_t d = tmem + (uint32_t)(slot * BN);
          const int kb0 = c * kb_per_chunk, kb1 = min(nkb, kb0 + kb_per_chunk);
          for (int kb = kb0; kb < kb1; ++kb, ++g) {
            const int s = g % S;
            if (!mbar_wait_bounded(full0 + 8 * s, (uint32_t)((g / S) & 1), kWaitBudgetCycles)) {
              ok = false;
              break;
            }
            tc_fence_after();
#pragma unroll
            for (int k16 = 0; k16 < kBK / 16; ++k16) {
              const uint64_t ad = sdesc_swz(sA + (uint32_t)s * kABytes + 32u * k16);
              const uint64_t bd = sdesc_swz(sB + (uint32_t)s * GG::BBytes + 32u * k16);
              tc_mma(d, ad, bd, idesc, (kb == kb0 && k16 == 0) ? 0u : 1u);
            }
            tc_commit(empty0 + 8 * s);
          }
          if (ok) tc_commit(accf0 + 8 * slot);
        }
      }
      if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
      tc_commit(done);  // completes once every MMA issued above has completed
      if (!mbar_wait_bounded(done, 0u, kWaitBudgetCycles)) atomicOr(a.err, DEVERR_DRAIN_WAIT);
    }
  } else {
    // ---------------------------------------------------------------------- epilogue warps 0-3
    const uint32_t lane_base = tmem + ((uint32_t)(32 * warp) << 16);
    const bool want_top = a.kind == EPI_F32 && a.top1 != nullptr;
    bool ok = true;
    int q = 0;
    for (int t = blockIdx.x; t < tiles && ok; t += gridDim.x) {
      const int n0 = (t % NT) * BN, m0 = (t / NT) * kBM;
      const int row = m0 + 32 * warp + lane;
      unsigned long long best = 0ull;
      // the epilogue of 32 consecutive columns c0 .. c0+31 of this thread's row
      auto emit32 = [&](int c0, const float (&v)[32]) {
        if (row >= a.M) return;
        const int col0 = n0 + c0;
        if (a.kind == EPI_GEGLU) {
#pragma unroll
          for (int hq = 0; hq < 2; ++hq) {  // two 16-column blocks: gate 0..7, up 8..15
            const int cb = col0 + 16 * hq;
            if (cb + 16 > a.N) continue;
            float h[8];
#pragma unroll
            for (int j = 0; j < 8; ++j) h[j] = geglu_recipe(v[16 * hq + j], v[16 * hq + 8 + j]);
            uint4 w;
            w.x = pack_bf16x2(h[0], h[1]);
            w.y = pack_bf16x2(h[2], h[3]);
            w.z = pack_bf16x2(h[4], h[5]);
            w.w = pack_bf16x2(h[6], h[7]);
            *reinterpret_cast<uint4*>(a.y + (size_t)row * (a.N >> 1) + (cb >> 1)) = w;
          }
        } else if (a.kind == EPI_BF16) {
#pragma unroll
          for (int j8 = 0; j8 < 4; ++j8) {
            const int cb = col0 + 8 * j8;
            if (cb + 8 <= a.N) {
              uint4 w;
              w.x = pack_bf16x2(v[8 * j8 + 0], v[8 * j8 + 1]);
              w.y = pack_bf16x2(v[8 * j8 + 2], v[8 * j8 + 3]);
              w.z = pack_bf16x2(v[8 * j8 + 4], v[8 * j8 + 5]);
              w.w = pack_bf16x2(v[8 * j8 + 6], v[8 * j8 + 7]);
              *reinterpret_cast<uint4*>(a.y + (size_t)row * a.N + cb) = w;
            }
          }
        } else {
#pragma unroll
          for (int j4 = 0; j4 < 8; ++j4) {
            const int cb = col0 + 4 * j4;
            if (cb + 4 <= a.N && a.logits)
              *reinterpret_cast<float4*>(a.logits + (size_t)row * a.N + cb) =
                  make_float4(v[4 * j4], v[4 * j4 + 1], v[4 * j4 + 2], v[4 * j4 + 3]);
          }
          if (want_top) {
#pragma unroll
            for (int j = 0; j < 32; ++j) {
              const int col = col0 + j;
              if (col < a.N) {
                const unsigned long long key = ((unsigned long long)float_order_key(v[j]) << 32) |
                                               (unsigned long long)(0xFFFFFFFFu - (uint32_t)col);
                best = key > best ? key : best;
              }
            }
          }
        }
      };
      if constexpr (kInt8) {
        int isum[BN];
#pragma unroll
        for (int j = 0; j < BN; ++j) isum[j] = 0;
        for (int c = 0; c < nchunks; ++c, ++q) {
          const int slot = q % NSLOT;
          if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
            ok = false;
            atomicOr(a.err, DEVERR_CONSUMER_WAIT);
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int g = 0; g < BN / 32; ++g) {
            uint32_t r[32];
            tmem_ld32(lane_base + (uint32_t)(slot * BN + 32 * g), r);
#pragma unroll
            for (int j = 0; j < 32; ++j) isum[32 * g + j] += __float2int_rn(__uint_as_float(r[j]));
          }
          tc_fence_before();
          mbar_arrive(acce0 + 8 * slot);
        }
        if (!ok) break;
        const float sx = row < a.M ? a.s_x[row] : 0.0f;
#pragma unroll
        for (int g = 0; g < BN / 32; ++g) {
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int col = n0 + 32 * g + j;
            float y = 0.0f;
            if (col < a.N) {
              y = __fmul_rn(__fmul_rn(sx, a.s_w[col]), __int2float_rn(isum[32 * g + j]));
              if (a.bias) y = __fadd_rn(y, a.bias[col]);
              if (a.acc_dbg && row < a.M) a.acc_dbg[(size_t)row * a.N + col] = isum[32 * g + j];
            }
            v[j] = y;
          }
          emit32(32 * g, v);
        }
      } else {
        const int slot = q % NSLOT;
        if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
          ok = false;
          atomicOr(a.err, DEVERR_CONSUMER_WAIT);
          break;
        }
        tc_fence_after();
#pragma unroll 1
        for (int g = 0; g < BN / 32; ++g) {
          uint32_t r[32];
          tmem_ld32(lane_base + (uint32_t)(slot * BN + 32 * g), r);
          float v[32];
#pragma unroll
          for (int j = 0; j < 32; ++j) {
            const int col = n0 + 32 * g + j;
            float y = __uint_as_float(r[j]);
            if (a.bias && col < a.N) y = __fadd_rn(y, a.bias[col]);
            v[j] = y;
          }
          emit32(32 * g, v);
        }
        tc_fence_before();
        mbar_arrive(acce0 + 8 * slot);
        ++q;
      }
      if (want_top && row < a.M && best != 0ull) atomicMax(a.top_keys + row, best);
    }
    // top-1 across the grid: the last CTA to finish decodes the per-row keys and clears them
    if (want_top) {
      __threadfence();
      named_bar_sync(1, 128);
      if (threadIdx.x == 0) {
        const unsigned int prev = atomicAdd(a.grid_counter, 1u);
        s_flag = prev == gridDim.x - 1;
        if (s_flag) *a.grid_counter = 0u;
      }
      named_bar_sync(1, 128);
      if (s_flag) {
        __threadfence();
        for (int t = threadIdx.x; t < a.M; t += 128) {
          const unsigned long long key = atomicExch(a.top_keys + t, 0ull);
          a.top1[t] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == 5) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

template <bool kInt8, int kBN>
w8a8_status launch_t(const TcArgs& a, cudaStream_t st) {
  using GG = TcGeo<kInt8, kBN>;
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(gemm_tc_kernel<kInt8, kBN>, cudaFuncAttributeMaxDynamicSharedMemorySize, GG::Smem));
    attr_set[dev] = true;
  }
  CUtensorMap ta, tb;
  W8A8_TRY(make_tmap_2d(&ta, a.A, 2, (uint64_t)a.K, (uint64_t)a.M, (uint64_t)a.K * 2, kBK, kBM, kSwz));
  W8A8_TRY(make_tmap_2d(&tb, a.B, 2, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K * 2, kBK, GG::BN, kSwz));
  const long long tiles = (long long)((a.N + GG::BN - 1) / GG::BN) * ((a.M + kBM - 1) / kBM);
  const dim3 grid((unsigned)std::min<long long>(tiles, device_sms()));
  W8A8_CUDA(launch_pdl(gemm_tc_kernel<kInt8, kBN>, grid, dim3(kThreads), (size_t)GG::Smem, st, ta, tb, a));
  return W8A8_OK;
}

}  // namespace

bool tc_gemm_supported(int M, int N, int K, int kind, bool want_top, int max_top) {
  if (M < 1 || N < 16 || K < 16 || K % 16 != 0 || N % 16 != 0) return false;
  if (kind != EPI_BF16 && kind != EPI_GEGLU && kind != EPI_F32) return false;
  if (want_top && M > max_top) return false;
  return true;
}

w8a8_status launch_tc_gemm(bool int8_codes, const TcArgs& a, cudaStream_t st) {
  if (a.M == 0 || a.N == 0) return W8A8_OK;
  void *v0, *v1;
  take_kernel_events(&v0, &v1);
  cudaEvent_t e0 = reinterpret_cast<cudaEvent_t>(v0), e1 = reinterpret_cast<cudaEvent_t>(v1);
  if (e0) W8A8_CUDA(cudaEventRecord(e0, st));
  // bf16: 256-channel tiles unless that leaves SMs without a tile
  const long long tiles256 = (long long)((a.N + 255) / 256) * ((a.M + kBM - 1) / kBM);
  const w8a8_status s = int8_codes                    ? launch_t<true, 128>(a, st)
                        : tiles256 >= device_sms() ? launch_t<false, 256>(a, st)
                                                   : launch_t<false, 128>(a, st);
  if (e1) W8A8_CUDA(cudaEventRecord(e1, st));
  return s;
}

}  // namespace w8a8
