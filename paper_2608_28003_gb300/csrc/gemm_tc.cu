// Tensor-core GEMM (tcgen05, TMEM accumulators, TMA) for prefill-sized token counts.
//
// A persistent grid (one CTA per SM) walks the output tiles of 128 tokens x BN channels.  A
// (tokens x K) and B (channels x K) tiles of 64 k arrive by 2-D TMA into 128-byte-swizzled shared
// memory, S stages deep, continuously across tiles.  Accumulators live in tensor memory (all 512
// columns), as a ring of slots (BN rounded up to 128 or 256 columns), so the epilogue of one tile
// overlaps the MMAs of the next.
//  * warp 16 (one thread) issues the TMA copies; warp 17 allocates tensor memory and one of its
//    threads issues tcgen05.mma (M = 128, N = BN, K = 16, fp32 accumulation) for each stage,
//    commits the stage back to the producer and each finished slot to the epilogue; warps 0-15 are
//    the epilogue, warp w reading TMEM lanes 32 (w mod 4) .. +31 (its tokens) and column quarter
//    w / 4 of the slot with tcgen05.ld, then handing the slot back.  Four epilogue warps per SM
//    sub-partition keep its issue slots busy while one waits on a dependency.
//  * tiles: BN = 64 / 128 (four slots) on single CTAs, or BN = 192 / 256 (two slots) on CTA pairs
//    of 256 tokens (cta_group::2, below), chosen by a cost model of the waves.
//  * W8A8 path: both operands are INT8 codes stored as fp16 (exact).  Every product is an integer
//    below 2^14, so a fp32 sum of at most 1024 of them is exact; the accumulator is therefore
//    restarted every 1024 k (16 stages) in the next slot while the epilogue folds the finished one
//    into INT32 registers, and the INT32 result is exact in any order (Eq. gemm-final).  The
//    epilogue then dequantises fl(fl(s_x s_w) acc) (+ bias).
//  * bf16 path: one accumulator per tile over the whole k range.
//  * FP8 path (the e4m3 variant of the W8A8 linear): both operands are e4m3 codes, one byte each;
//    tcgen05.mma kind::f8f6f4 (K = 32 per instruction) reads the same 128-byte swizzled rows, so a
//    stage carries 128 k in the bytes a fp16 stage uses for 64, and the fp32 accumulator runs over
//    the whole k range (fp32 sums of e4m3 products are not exact; no fold) before the epilogue
//    dequantises fl(fl(s_x s_w) acc).
//  * epilogues: bf16 output, GeGLU of interleaved gate/up columns (16-column blocks: 8 gate, then
//    the 8 matching up channels), or fp32 logits with the top-1 index (keys reduced with atomicMax,
//    the last CTA to finish decodes them); outputs leave through 32 x 32 shared-memory blocks and
//    2-D TMA stores.
// Every mbarrier wait is bounded: on timeout the kernel sets a bit of the error word, stops, waits
// (bounded) for its own copies and MMAs in flight and frees its tensor memory.
#include <algorithm>

#include "gemm_tc.cuh"
#include "tc_common.cuh"
#include "ops.cuh"
#include "stream_gemm.cuh"
#include "tmap.cuh"

namespace w8a8 {

namespace {

constexpr int kBM = 128;
constexpr int kSwz = kTcSwz;             // swizzle span in bytes (TMA and the MMA descriptors agree)
constexpr int kBK = kSwz / 2;            // k per stage: one swizzle span of fp16 per row
// operand modes: bf16 pass-through, INT8 codes carried as fp16 (exact, folded), e4m3 codes
constexpr int kModeBf16 = TC_BF16, kModeI8 = TC_I8, kModeFp8 = TC_FP8;
// k elements per stage: one 128-byte swizzle span per row (64 two-byte or 128 one-byte elements)
__host__ __device__ constexpr int bk_elems(int mode) { return mode == kModeFp8 ? kSwz : kSwz / 2; }
__host__ __device__ constexpr int elem_bytes(int mode) { return mode == kModeFp8 ? 1 : 2; }
constexpr int kEpiWarps = 16;                   // four per TMEM lane quarter: one per column quarter
constexpr int kParts = kEpiWarps / 4;
constexpr int kProdWarp = kEpiWarps, kMmaWarp = kEpiWarps + 1;
constexpr int kThreads = 32 * (kEpiWarps + 2);
// The 512 epilogue threads test the rows once per kernel, while the first stages load: bit i of
// *fail is set when row tile i (rows_per_tile tokens) has a token past the bound.  Row tiles past
// the 32nd always take the chunked path.  Ends with the epilogue warps' named barrier 3; the
// first thread then arrives on the MMA issuer's barrier.
__device__ __forceinline__ void scan_exact(const TcArgs& a, int rows_per_tile, uint32_t* fail, uint32_t ready) {
  const int rows = min(a.M, 32 * rows_per_tile);
  uint32_t f = 0u;
  for (int i = threadIdx.x; i < rows; i += 32 * kEpiWarps)
    if (__ldg(a.qsum + i) > kExactQsum) f |= 1u << (i / rows_per_tile);
  f = __reduce_or_sync(0xffffffffu, f);
  if ((threadIdx.x & 31) == 0 && f) atomicOr(fail, f);
  named_bar_sync(3, 32 * kEpiWarps);
  if (threadIdx.x == 0) mbar_arrive(ready);
}
__device__ __forceinline__ bool row_tile_exact(uint32_t fail, int i) { return i < 32 && !((fail >> i) & 1u); }
constexpr uint32_t kTmemCols = 512;  // all of an SM's tensor memory: 2 (bf16) or 4 (W8A8) accumulator slots
constexpr uint32_t kABytes = kBM * kBK * 2;
constexpr int kStageBufBytes = 32 * 64;                  // one epilogue block: 32 rows of 64 bytes
constexpr int kEpiSmem = kEpiWarps * kStageBufBytes;  // one block per epilogue warp

// Rows of the activation box a stage loads: with fewer than 128 tokens only the rows that exist
// (rounded up to 8) are copied; the MMA still reads 128 rows, but rows past M only feed output
// rows that are never stored, so the rest of the tile is left as it is (a zero fill would cost as
// much TMA time as real data).
__host__ __device__ constexpr int a_box_rows(int M) { return M < kBM ? (M + 7) / 8 * 8 : kBM; }

// Tensor-memory columns of one accumulator slot: BN rounded up to a power of two, so every slot
// starts on a 128-column boundary.
__host__ __device__ constexpr int slot_cols(int bn) { return bn <= 128 ? 128 : bn <= 256 ? 256 : 512; }

template <int kMode, int kBN>
struct TcGeo {
  static constexpr int BN = kBN;
  static constexpr uint32_t BBytes = BN * kBK * 2;
  static constexpr int S = (192 * 1024) / (int)(kABytes + BBytes);
  static constexpr int Smem = S * (kABytes + BBytes) + kEpiSmem + 1024;
};

// ---------------------------------------------------------------------------- tcgen05 helpers
template <int kMode>
__device__ __forceinline__ void tc_mma_m(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                         uint32_t accumulate) {
  if constexpr (kMode == kModeFp8)
    tc_mma_f8(d_tmem, a_desc, b_desc, idesc, accumulate);
  else
    tc_mma(d_tmem, a_desc, b_desc, idesc, accumulate);
}
// Two fp32 values -> bf16x2 (a in the low half), each rounded to nearest even: one instruction.
__device__ __forceinline__ uint32_t pack_bf16x2(float a, float b) {
  uint32_t r;
  asm("cvt.rn.bf16x2.f32 %0, %1, %2;\n" : "=r"(r) : "f"(b), "f"(a));
  return r;
}

// 32 consecutive fp32 values p[c0 .. c0 + 31] into w, 0 past n (c0 a multiple of 32, p 16-byte
// aligned): eight 16-byte loads when the group lies inside n.  Every lane of a warp reads the same
// addresses (a broadcast).

// The dequantising epilogue of one 32-column group: w holds s_w of the columns on entry and
// fl(fl(s_x s_w) acc) (+ bias) on exit (Eq. gemm-final); acc is the INT32 sum (W8A8) or the fp32
// one (FP8).
template <typename T>
__device__ __forceinline__ float acc_as_f32(T v);
template <>
__device__ __forceinline__ float acc_as_f32<int>(int v) { return __int2float_rn(v); }
template <>
__device__ __forceinline__ float acc_as_f32<uint32_t>(uint32_t v) { return __uint_as_float(v); }

// Column values of the epilogue (s_w, bias) one column per lane: lane j holds column c0 + j of
// each of the warp's NG groups, loaded at the start of a tile, before the wait for its
// accumulator, so that the load latency overlaps the MMAs; element j of a group takes its values
// from lane j with a shuffle.
template <int NG>
struct ColVals {
  float sw[NG], b[NG];
};
template <int NG>
__device__ __forceinline__ void load_colvals(const TcArgs& a, bool want_sw, int n0, int part, int bn, int lane,
                                             ColVals<NG>& cv) {
#pragma unroll
  for (int i = 0; i < NG; ++i) {
    const int c = n0 + 32 * (part + kParts * i) + lane;
    const bool in = 32 * (part + kParts * i) < bn && c < a.N;
    cv.sw[i] = want_sw && in ? __ldg(a.s_w + c) : 0.0f;
    cv.b[i] = a.bias && in ? __ldg(a.bias + c) : 0.0f;
  }
}
// fl(fl(s_x s_w) acc) (+ bias) of one 32-column group (Eq. gemm-final); acc is the INT32 sum
// (W8A8) or the fp32 one (FP8); sw / b are this lane's column values of the group.
// Two IEEE fp32 products, each rounded to nearest even (the packed form of two __fmul_rn).
__device__ __forceinline__ void fmul2_rn(float a0, float a1, float b0, float b1, float& d0, float& d1) {
  const unsigned long long x = ((unsigned long long)__float_as_uint(a1) << 32) | __float_as_uint(a0);
  const unsigned long long y = ((unsigned long long)__float_as_uint(b1) << 32) | __float_as_uint(b0);
  unsigned long long z;
  asm("mul.rn.f32x2 %0, %1, %2;\n" : "=l"(z) : "l"(x), "l"(y));
  d0 = __uint_as_float((uint32_t)z);
  d1 = __uint_as_float((uint32_t)(z >> 32));
}
template <typename T>
__device__ __forceinline__ void dequant32(bool has_bias, float sx, float sw, float b, const T* acc, float (&v)[32]) {
#pragma unroll
  for (int j = 0; j < 32; j += 2) {
    float t0, t1;
    fmul2_rn(sx, sx, __shfl_sync(0xffffffffu, sw, j), __shfl_sync(0xffffffffu, sw, j + 1), t0, t1);
    fmul2_rn(t0, t1, acc_as_f32<T>(acc[j]), acc_as_f32<T>(acc[j + 1]), v[j], v[j + 1]);
    if (has_bias) {
      v[j] = __fadd_rn(v[j], __shfl_sync(0xffffffffu, b, j));
      v[j + 1] = __fadd_rn(v[j + 1], __shfl_sync(0xffffffffu, b, j + 1));
    }
  }
}
__device__ __forceinline__ void add_bias32(float b, float (&v)[32]) {
#pragma unroll
  for (int j = 0; j < 32; ++j) v[j] = __fadd_rn(v[j], __shfl_sync(0xffffffffu, b, j));
}

// ------------------------------------------------------------------ epilogue through TMA stores
// Each epilogue warp stages 32 rows x 32 columns of output (its rows, one 32-column group) in its
// 2 KB shared-memory block and one lane stores the block with a 2-D TMA store (rows past M and
// columns past N are clipped by the tensor map), so the global writes are whole rows, not one
// 16-byte piece per thread and row; the warp waits for the store to have read the block before it
// refills it (the other warps of its sub-partition issue meanwhile).  A staged row is 64 bytes (32 bf16 or 16 fp32: fp32 output goes
// out as two blocks of 16 columns) or 32 (GeGLU); the block is kept in the tensor map's swizzled
// layout of that width (16-byte chunk c of row r at chunk c ^ ((r >> 1) & 3), or c ^ ((r >> 2) & 1)),
// so the 16-byte stores of eight consecutive rows fall in eight different bank groups.

__device__ __forceinline__ void fence_proxy_async_shared() {
  asm volatile("fence.proxy.async.shared::cta;\n" ::: "memory");
}
__device__ __forceinline__ void tma_store_2d(const void* tmap, uint32_t src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];\n" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(src), "r"(c0), "r"(c1)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_read0() { asm volatile("cp.async.bulk.wait_group.read 0;\n" ::: "memory"); }
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;\n" ::: "memory"); }

// The epilogue of 32 consecutive columns col0 .. col0+31 of this thread's row (lane of the warp
// whose rows start at row0): bf16 output, GeGLU of the interleaved gate/up columns (two 16-column
// blocks: 8 gate, then the 8 matching up channels), or fp32 logits with the row's running top-1 key.
__device__ __forceinline__ void stage_cols32(const TcArgs& a, const CUtensorMap* tmY, uint32_t buf,
                                             int row0, int col0, int lane, const float (&v)[32], bool want_top,
                                             unsigned long long& best) {
  const int row = row0 + lane;
  if (a.kind == EPI_F32 && want_top && row < a.M) {
#pragma unroll
    for (int j = 0; j < 32; ++j) {
      const int col = col0 + j;
      if (col < a.N) {
        const unsigned long long key =
            ((unsigned long long)float_order_key(v[j]) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)col);
        best = key > best ? key : best;
      }
    }
  }
  if (a.kind == EPI_F32) {
    if (!a.logits) return;  // top-1 only
#pragma unroll
    for (int h = 0; h < 2; ++h) {
      if (lane == 0) bulk_wait_read0();  // the previous store has read the block
      __syncwarp();
      const uint32_t dst = buf + (uint32_t)(lane * 64), sw = (uint32_t)((lane >> 1) & 3);
#pragma unroll
      for (int j4 = 0; j4 < 4; ++j4)
        asm volatile("st.shared.v4.f32 [%0], {%1, %2, %3, %4};\n" ::"r"(dst + 16 * ((uint32_t)j4 ^ sw)),
                     "f"(v[16 * h + 4 * j4]), "f"(v[16 * h + 4 * j4 + 1]), "f"(v[16 * h + 4 * j4 + 2]),
                     "f"(v[16 * h + 4 * j4 + 3])
                     : "memory");
      fence_proxy_async_shared();
      __syncwarp();
      if (lane == 0) {
        tma_store_2d(tmY, buf, col0 + 16 * h, row0);
        bulk_commit();
      }
    }
    return;
  }
  if (lane == 0) bulk_wait_read0();  // the previous store has read the block
  __syncwarp();
  if (a.kind == EPI_GEGLU) {
    uint32_t w[8];
#pragma unroll
    for (int hq = 0; hq < 2; ++hq)
#pragma unroll
      for (int j = 0; j < 8; j += 2)
        w[4 * hq + j / 2] = pack_bf16x2(geglu_recipe(v[16 * hq + j], v[16 * hq + 8 + j]),
                                        geglu_recipe(v[16 * hq + j + 1], v[16 * hq + 9 + j]));
    const uint32_t dst = buf + (uint32_t)(lane * 32), sw = (uint32_t)((lane >> 2) & 1);
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};\n" ::"r"(dst + 16 * sw), "r"(w[0]), "r"(w[1]), "r"(w[2]),
                 "r"(w[3])
                 : "memory");
    asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};\n" ::"r"(dst + 16 * (1u ^ sw)), "r"(w[4]), "r"(w[5]),
                 "r"(w[6]), "r"(w[7])
                 : "memory");
  } else {
    const uint32_t dst = buf + (uint32_t)(lane * 64), sw = (uint32_t)((lane >> 1) & 3);
#pragma unroll
    for (int j8 = 0; j8 < 4; ++j8)
      asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};\n" ::"r"(dst + 16 * ((uint32_t)j8 ^ sw)),
                   "r"(pack_bf16x2(v[8 * j8], v[8 * j8 + 1])), "r"(pack_bf16x2(v[8 * j8 + 2], v[8 * j8 + 3])),
                   "r"(pack_bf16x2(v[8 * j8 + 4], v[8 * j8 + 5])), "r"(pack_bf16x2(v[8 * j8 + 6], v[8 * j8 + 7]))
                   : "memory");
  }
  fence_proxy_async_shared();
  __syncwarp();
  if (lane == 0) {
    tma_store_2d(tmY, buf, a.kind == EPI_GEGLU ? col0 >> 1 : col0, row0);
    bulk_commit();
  }
}

// The last unit of a split tile: the 512 epilogue threads sum the tile's KS partials (units u0 ..
// u0 + KS - 1) in part order, four columns per thread with every part's load in flight, and write
// the bf16 outputs (W8A8: the INT32 sums dequantised exactly as the tile epilogue does it).
template <int kMode, int BN>
__device__ __forceinline__ void split_reduce(const TcArgs& a, int u0, int KS, int R, int m0, int n0) {
  const uint4* part = reinterpret_cast<const uint4*>(a.partials) + (size_t)u0 * R * (BN / 4);
  const size_t pstride = (size_t)R * (BN / 4);
  for (int e = threadIdx.x; e < R * (BN / 4); e += 32 * kEpiWarps) {
    const int r = e / (BN / 4), c = 4 * (e % (BN / 4));
    const int row = m0 + r, col = n0 + c;
    if (row >= a.M || col >= a.N) continue;  // N is a multiple of 16: four columns are all in or out
    const uint4* p = part + e;
    float y[4];
    if constexpr (kMode == kModeI8) {
      int s[4] = {0, 0, 0, 0};
#pragma unroll 8
      for (int sp = 0; sp < KS; ++sp) {
        const uint4 v = __ldcg(p + sp * pstride);
        s[0] += (int)v.x;
        s[1] += (int)v.y;
        s[2] += (int)v.z;
        s[3] += (int)v.w;
      }
      const float sx = a.s_x[row];
#pragma unroll
      for (int k = 0; k < 4; ++k) y[k] = __fmul_rn(__fmul_rn(sx, a.s_w[col + k]), __int2float_rn(s[k]));
      if (a.acc_dbg)
        *reinterpret_cast<int4*>(a.acc_dbg + (size_t)row * a.N + col) = make_int4(s[0], s[1], s[2], s[3]);
    } else {
      y[0] = y[1] = y[2] = y[3] = 0.0f;
#pragma unroll 8
      for (int sp = 0; sp < KS; ++sp) {
        const uint4 v = __ldcg(p + sp * pstride);
        y[0] = __fadd_rn(y[0], __uint_as_float(v.x));
        y[1] = __fadd_rn(y[1], __uint_as_float(v.y));
        y[2] = __fadd_rn(y[2], __uint_as_float(v.z));
        y[3] = __fadd_rn(y[3], __uint_as_float(v.w));
      }
      if constexpr (kMode == kModeFp8) {  // the fp32 sum of all parts, dequantised
        const float sx = a.s_x[row];
#pragma unroll
        for (int k = 0; k < 4; ++k) y[k] = __fmul_rn(__fmul_rn(sx, a.s_w[col + k]), y[k]);
      }
    }
    if (a.bias) {
#pragma unroll
      for (int k = 0; k < 4; ++k) y[k] = __fadd_rn(y[k], a.bias[col + k]);
    }
    *reinterpret_cast<uint2*>(a.y + (size_t)row * a.N + col) = make_uint2(pack_bf16x2(y[0], y[1]), pack_bf16x2(y[2], y[3]));
  }
}

template <int kMode, int kBN>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tc_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmY, const TcArgs a) {
  using GG = TcGeo<kMode, kBN>;
  constexpr bool kInt8 = kMode == kModeI8, kFp8 = kMode == kModeFp8;
  constexpr int BKe = bk_elems(kMode);
  constexpr int BN = GG::BN, S = GG::S;
  constexpr int SC = slot_cols(BN), NSLOT = (int)kTmemCols / SC;  // accumulator slots in tensor memory
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t bars[2 * S + 2 * NSLOT + 2];
  __shared__ uint32_t tmem_slot;
  __shared__ int s_flag, s_last;
  __shared__ uint32_t s_fail;  // W8A8: row tiles with a token past the exactness bound

  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t sA = base, sB = base + (uint32_t)S * kABytes, stg = sB + (uint32_t)S * GG::BBytes;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int NT = (a.N + BN - 1) / BN, tiles = NT * ((a.M + kBM - 1) / kBM);
  const int nkb = (a.K + BKe - 1) / BKe;
  // work units: (tile, k part); unit u is part u mod KS of tile u / KS, stages [kb_lo, kb_hi)
  const int KS = a.ksplit > 1 ? a.ksplit : 1, units = tiles * KS;
  auto kb_lo = [&](int u) { return (int)((long long)(u % KS) * nkb / KS); };
  auto kb_hi = [&](int u) { return (int)((long long)(u % KS + 1) * nkb / KS); };
  // accumulator chunks of a unit (warp-collective): W8A8 restarts every chunk_stages(len) stages
  // (at most 1024 k) counted from the unit's first stage, unless the tile's tokens pass the
  // exactness bound (one chunk)
  // W8A8 row tiles are tested against the exactness bound when a tile's k range is not split (split
  // units are short: their first fold boundary would come before the scan ends) and spans more than
  // one chunk
  const bool scan = kInt8 && a.qsum != nullptr && KS == 1 && nkb > kKbPerChunk;
  auto unit_chunks = [&](int u) {  // epilogue side, after the scan
    const int n = kInt8 ? chunk_count(kb_hi(u) - kb_lo(u)) : 1;
    return n > 1 && !(scan && row_tile_exact(s_fail, (u / KS) / NT)) ? n : 1;
  };
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, accf0 = full0 + 16 * S, acce0 = accf0 + 8 * NSLOT,
                 done = acce0 + 8 * NSLOT, ready = done + 8;

  pdl_trigger();
  if (warp == kProdWarp && lane == 0) {
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    prefetch_tmap(&tmY);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < NSLOT; ++b) {
      mbar_init(accf0 + 8 * b, 1);
      mbar_init(acce0 + 8 * b, 32 * kEpiWarps);
    }
    mbar_init(done, 1);
    mbar_init(ready, 1);
    s_fail = 0u;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
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

  // Persistent: CTA b takes units b, b + grid, ...; tile t covers channels (t mod NT) * BN and
  // tokens (t / NT) * 128, so neighbouring CTAs share the activation rows.
  if (warp == kProdWarp) {
    // ---------------------------------------------------------------------- TMA producer
    if (lane == 0) {
      bool ok = true;
      int g = 0;  // stages issued
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        const int t = u / KS, n0 = (t % NT) * BN, m0 = (t / NT) * kBM;
        const int kb_end = kb_hi(u);
        for (int kb = kb_lo(u); kb < kb_end; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait_bounded(empty0 + 8 * s, (uint32_t)(((g / S) & 1) ^ 1), kWaitBudgetCycles)) {
            ok = false;
            break;
          }
          const uint32_t bar = full0 + 8 * s;
          mbar_arrive_expect_tx(bar, (uint32_t)(a_box_rows(a.M) * kSwz) + GG::BBytes);
          tma_load_2d(sA + (uint32_t)s * kABytes, &tmA, kb * BKe, m0, bar);
          tma_load_2d(sB + (uint32_t)s * GG::BBytes, &tmB, kb * BKe, n0, bar);
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
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------------- MMA issuer
    if (lane == 0) {
      constexpr uint32_t idesc = idesc_f16(kMode == kModeBf16 ? 1u : 0u, BN, kBM);
      bool ok = true, known = false;  // known: the epilogue's exactness scan has been read
      uint32_t fail = 0u;
      int g = 0, q = 0;  // stages consumed, accumulator chunks produced
      // One accumulator slot per chunk; a W8A8 unit restarts in the next slot at each fold boundary
      // (every chunk_stages(len) stages) unless its row tile passed the exactness bound, which is
      // first needed at the first boundary, when the scan has long finished.
      for (int u = blockIdx.x; u < units && ok; u += gridDim.x) {
        const int ulo = kb_lo(u), uhi = kb_hi(u), per = kInt8 ? chunk_stages(uhi - ulo) : uhi - ulo;
        int slot = q % NSLOT, kb0 = ulo, next_fold = ulo + per;
        if (q >= NSLOT &&  // the epilogue has drained this slot's previous chunk
            !mbar_wait_bounded(acce0 + 8 * slot, (uint32_t)(((q / NSLOT) - 1) & 1), kWaitBudgetCycles)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t d = tmem + (uint32_t)(slot * SC);
        for (int kb = ulo; kb < uhi; ++kb, ++g) {
          if (kInt8 && kb == next_fold) {  // a fold boundary
            next_fold += per;
            if (scan && !known) {
              if (!mbar_wait_bounded(ready, 0u, kWaitBudgetCycles)) {
                ok = false;
                break;
              }
              fail = s_fail;
              known = true;
            }
            if (!(scan && row_tile_exact(fail, (u / KS) / NT))) {
              tc_commit(accf0 + 8 * slot);
              ++q;
              slot = q % NSLOT;
              if (q >= NSLOT &&
                  !mbar_wait_bounded(acce0 + 8 * slot, (uint32_t)(((q / NSLOT) - 1) & 1), kWaitBudgetCycles)) {
                ok = false;
                break;
              }
              tc_fence_after();
              d = tmem + (uint32_t)(slot * SC);
              kb0 = kb;
            }
          }
          const int s = g % S;
          if (!mbar_wait_bounded(full0 + 8 * s, (uint32_t)((g / S) & 1), kWaitBudgetCycles)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int k16 = 0; k16 < kSwz / 32; ++k16) {  // 32 bytes of k per instruction
            const uint64_t ad = sdesc_swz(sA + (uint32_t)s * kABytes + 32u * k16);
            const uint64_t bd = sdesc_swz(sB + (uint32_t)s * GG::BBytes + 32u * k16);
            tc_mma_m<kMode>(d, ad, bd, idesc, (kb == kb0 && k16 == 0) ? 0u : 1u);
          }
          tc_commit(empty0 + 8 * s);
        }
        if (ok) tc_commit(accf0 + 8 * slot);
        ++q;
      }
      if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
      tc_commit(done);  // completes once every MMA issued above has completed
      if (!mbar_wait_bounded(done, 0u, kWaitBudgetCycles)) atomicOr(a.err, DEVERR_DRAIN_WAIT);
    }
  } else {
    // ---------------------------------------------------------------------- epilogue warps 0-15
    if (scan) scan_exact(a, kBM, &s_fail, ready);
    const int quad = warp & 3, part = warp >> 2;  // TMEM lane quarter (tokens), column quarter
    const uint32_t lane_base = tmem + ((uint32_t)(32 * quad) << 16);
    const bool want_top = a.kind == EPI_F32 && a.top1 != nullptr;
    const uint32_t buf = stg + (uint32_t)(warp * kStageBufBytes);
    bool ok = true;
    int q = 0;
    // split-K partials (bf16 outputs only): unit u's block of R rows x BN columns, row-major; a
    // thread stores its row's 32 sums of a column group as 16-byte vectors (W8A8: the INT32 sums,
    // bf16: the fp32 ones)
    const int R = a_box_rows(a.M), rloc = 32 * quad + lane;
    const bool has_row = rloc < R;
    auto store_part32 = [&](int u, int g, const uint32_t (&w)[32]) {
      uint32_t* p = reinterpret_cast<uint32_t*>(a.partials) + ((size_t)u * R + rloc) * BN + 32 * g;
#pragma unroll
      for (int k = 0; k < 8; ++k)
        __stcg(reinterpret_cast<uint4*>(p) + k, make_uint4(w[4 * k], w[4 * k + 1], w[4 * k + 2], w[4 * k + 3]));
    };
    for (int u = blockIdx.x; u < units; u += gridDim.x) {
      const int t = u / KS, n0 = (t % NT) * BN, m0 = (t / NT) * kBM;
      const int row = m0 + rloc;
      unsigned long long best = 0ull;
      auto emit32 = [&](int c0, const float (&v)[32]) {
        stage_cols32(a, &tmY, buf, m0 + 32 * quad, n0 + c0, lane, v, want_top, best);
      };
      // After this unit's partials are stored: true when the unit is the tile's last to arrive (it
      // then sums all parts in part order); false, or a failed wait anywhere in the epilogue, ends it.
      auto arrive_last = [&]() -> bool {
        __threadfence();
        if (!named_bar_all(2, 32 * kEpiWarps, ok)) {
          ok = false;
          return false;
        }
        if (threadIdx.x == 0) {
          const unsigned int prev = atomicAdd(a.tile_counters + t, 1u);
          s_last = prev == (unsigned int)(KS - 1);
          if (s_last) a.tile_counters[t] = 0u;
        }
        named_bar_sync(2, 32 * kEpiWarps);
        if (!s_last) return false;
        __threadfence();
        return true;
      };
      if constexpr (kInt8) {
        constexpr int NG = (BN / 32 + kParts - 1) / kParts;  // this warp's 32-column groups: part + kParts i
        int isum[32 * NG];
#pragma unroll
        for (int j = 0; j < 32 * NG; ++j) isum[j] = 0;
        const int nch = unit_chunks(u);
        ColVals<NG> cv;  // before the first wait: the loads overlap the MMAs
        if (KS == 1) load_colvals<NG>(a, true, n0, part, BN, lane, cv);
        const float sx = KS == 1 && row < a.M ? a.s_x[row] : 0.0f;
        if (nch == 1 && KS == 1) {  // one exact fp32 accumulator: the INT32 sum as a float
          const int slot = q % NSLOT;
          if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
            ok = false;
            atomicOr(a.err, DEVERR_CONSUMER_WAIT);
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int i = 0; i < NG; ++i) {
            const int g = part + kParts * i;
            if (g >= BN / 32) break;
            uint32_t r[32];
            tmem_ld32(lane_base + (uint32_t)(slot * SC + 32 * g), r);
            if (a.acc_dbg && row < a.M) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (n0 + 32 * g + j < a.N)
                  a.acc_dbg[(size_t)row * a.N + n0 + 32 * g + j] = __float2int_rn(__uint_as_float(r[j]));
            }
            float v[32];
            dequant32(a.bias != nullptr, sx, cv.sw[i], cv.b[i], r, v);
            emit32(32 * g, v);
          }
          tc_fence_before();
          mbar_arrive(acce0 + 8 * slot);
          ++q;
          if (want_top && row < a.M && best != 0ull) atomicMax(a.top_keys + row, best);
          continue;
        }
        for (int c = 0; c < nch; ++c, ++q) {
          const int slot = q % NSLOT;
          if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
            ok = false;
            atomicOr(a.err, DEVERR_CONSUMER_WAIT);
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int i = 0; i < NG; ++i) {
            const int g = part + kParts * i;
            if (g >= BN / 32) break;
            uint32_t r[32];
            tmem_ld32(lane_base + (uint32_t)(slot * SC + 32 * g), r);
#pragma unroll
            for (int j = 0; j < 32; ++j) isum[32 * i + j] += __float2int_rn(__uint_as_float(r[j]));
          }
          tc_fence_before();
          mbar_arrive(acce0 + 8 * slot);
        }
        if (KS > 1) {
          if (ok && has_row) {
#pragma unroll
            for (int i = 0; i < NG; ++i) {
              const int g = part + kParts * i;
              if (g >= BN / 32) break;
              store_part32(u, g, reinterpret_cast<const uint32_t(&)[32]>(isum[32 * i]));
            }
          }
          if (arrive_last()) split_reduce<kModeI8, BN>(a, t * KS, KS, R, m0, n0);
          if (!ok) break;
          continue;
        } else if (!ok) {
          break;
        }
#pragma unroll
        for (int i = 0; i < NG; ++i) {
          const int g = part + kParts * i;
          if (g >= BN / 32) break;
          if (a.acc_dbg && row < a.M) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (n0 + 32 * g + j < a.N) a.acc_dbg[(size_t)row * a.N + n0 + 32 * g + j] = isum[32 * i + j];
          }
          float v[32];
          dequant32(a.bias != nullptr, sx, cv.sw[i], cv.b[i], &isum[32 * i], v);
          emit32(32 * g, v);
        }
      } else {
        constexpr int NG = (BN / 32 + kParts - 1) / kParts;
        ColVals<NG> cv;  // before the wait: the loads overlap the MMAs
        if (KS == 1) load_colvals<NG>(a, kFp8, n0, part, BN, lane, cv);
        const float sx = kFp8 && KS == 1 && row < a.M ? a.s_x[row] : 0.0f;
        const int slot = q % NSLOT;
        if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
          ok = false;
          atomicOr(a.err, DEVERR_CONSUMER_WAIT);
        } else {
          tc_fence_after();
#pragma unroll
          for (int i = 0; i < NG; ++i) {
            const int g = part + kParts * i;
            if (g >= BN / 32) break;
            uint32_t r[32];
            tmem_ld32(lane_base + (uint32_t)(slot * SC + 32 * g), r);
            if (KS > 1) {  // this part's fp32 sums go to the partials
              if (has_row) store_part32(u, g, r);
              continue;
            }
            float v[32];
            if constexpr (kFp8) {
              dequant32(a.bias != nullptr, sx, cv.sw[i], cv.b[i], r, v);
            } else {
#pragma unroll
              for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
              if (a.bias) add_bias32(cv.b[i], v);
            }
            emit32(32 * g, v);
          }
          tc_fence_before();
          mbar_arrive(acce0 + 8 * slot);
        }
        ++q;
        if (KS > 1) {
          if (arrive_last()) split_reduce<kMode, BN>(a, t * KS, KS, R, m0, n0);
          if (!ok) break;
          continue;
        } else if (!ok) {
          break;
        }
      }
      if (want_top && row < a.M && best != 0ull) atomicMax(a.top_keys + row, best);
    }
    if (lane == 0) bulk_wait_all();  // this warp's output stores have completed
    __syncwarp();
    // top-1 across the grid: the last CTA to finish decodes the per-row keys and clears them
    if (want_top) {
      __threadfence();
      named_bar_sync(1, 32 * kEpiWarps);
      if (threadIdx.x == 0) {
        const unsigned int prev = atomicAdd(a.grid_counter, 1u);
        s_flag = prev == gridDim.x - 1;
        if (s_flag) *a.grid_counter = 0u;
      }
      named_bar_sync(1, 32 * kEpiWarps);
      if (s_flag) {
        __threadfence();
        for (int t = threadIdx.x; t < a.M; t += 32 * kEpiWarps) {
          const unsigned long long key = atomicExch(a.top_keys + t, 0ull);
          a.top1[t] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  if (warp == kMmaWarp) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

// ------------------------------------------------------------------------- 2-CTA variant
// The same GEMM on CTA pairs (clusters of 2) with tcgen05.mma.cta_group::2: a pair computes a tile
// of 256 tokens x BN channels; CTA r holds tokens m0 + 128 r .. +127 of A and channels
// n0 + r BN/2 .. + BN/2 - 1 of B in its shared memory, so each SM loads half of the B tile, and its
// tensor memory receives its 128 rows of D.  CTA 0 of the pair issues the MMAs; both CTAs' TMA
// copies complete on CTA 0's stage barrier; the stage and accumulator barriers of both CTAs are
// signalled by multicast commits; both CTAs' epilogue threads hand the slot back to CTA 0.
template <int kMode, int kBN>
struct Tc2Geo {
  static constexpr int BN = kBN;
  static constexpr uint32_t BHalf = (kBN / 2) * kBK * 2;
  static constexpr int S = (192 * 1024) / (int)(kABytes + BHalf);
  static constexpr int Smem = S * (kABytes + BHalf) + kEpiSmem + 1024;
};

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;\n" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;\n" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;\n" ::: "memory");
}
__device__ __forceinline__ uint32_t map_to_rank(uint32_t addr, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;\n" : "=r"(r) : "r"(addr), "r"(rank));
  return r;
}
__device__ __forceinline__ void mbar_arrive_cluster(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];\n" ::"r"(cluster_addr) : "memory");
}
// 2-D TMA load into this CTA's shared memory whose completion is counted on an mbarrier of either
// CTA of the pair (cluster address).
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const void* tmap, int c0, int c1, uint32_t bar_cluster) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], "
      "[%4];\n" ::"r"(dst),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(c0), "r"(c1), "r"(bar_cluster)
      : "memory");
}
__device__ __forceinline__ void tc2_mma(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                        uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc2_mma_f8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                           uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::2.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
template <int kMode>
__device__ __forceinline__ void tc2_mma_m(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  if constexpr (kMode == kModeFp8)
    tc2_mma_f8(d_tmem, a_desc, b_desc, idesc, accumulate);
  else
    tc2_mma(d_tmem, a_desc, b_desc, idesc, accumulate);
}
// arrive on the barrier at this shared-memory offset in both CTAs of the pair once the MMAs issued
// so far have completed
__device__ __forceinline__ void tc2_commit_both(uint32_t bar) {
  const uint16_t mask = 0x3;
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;\n" ::"r"(bar),
      "h"(mask)
      : "memory");
}
__device__ __forceinline__ void tc2_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar) : "memory");
}

template <int kMode, int kBN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    gemm_tc2_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                    const __grid_constant__ CUtensorMap tmY, const TcArgs a) {
  using GG = Tc2Geo<kMode, kBN>;
  constexpr bool kInt8 = kMode == kModeI8, kFp8 = kMode == kModeFp8;
  constexpr int BKe = bk_elems(kMode);
  constexpr int BN = GG::BN, S = GG::S;
  constexpr int SC = slot_cols(BN), NSLOT = (int)kTmemCols / SC;
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  __shared__ uint64_t bars[2 * S + 2 * NSLOT + 2];
  __shared__ uint32_t tmem_slot;
  __shared__ int s_flag;
  __shared__ uint32_t s_fail;  // W8A8: row tiles with a token past the exactness bound

  const uint32_t raw = smem_u32(smem_raw);
  const uint32_t base = (raw + 1023u) & ~1023u;
  const uint32_t sA = base, sB = base + (uint32_t)S * kABytes, stg = sB + (uint32_t)S * GG::BHalf;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t rank = cluster_rank();
  const int pair = blockIdx.x >> 1, npairs = gridDim.x >> 1;
  const int NT = (a.N + BN - 1) / BN, tiles = NT * ((a.M + 2 * kBM - 1) / (2 * kBM));
  const int nkb = (a.K + BKe - 1) / BKe;
  const int nchunks = kInt8 ? chunk_count(nkb) : 1;
  const int kb_per_chunk = kInt8 ? chunk_stages(nkb) : nkb;
  // accumulator chunks of tile t (warp-collective): one where its 256 tokens pass the exactness bound
  // W8A8 row tiles (256 tokens) are tested against the exactness bound when K spans several chunks
  const bool scan = kInt8 && a.qsum != nullptr && nchunks > 1;
  auto tile_chunks = [&](int t) {  // epilogue side, after the scan
    return nchunks > 1 && !(scan && row_tile_exact(s_fail, t / NT)) ? nchunks : 1;
  };
  const uint32_t full0 = smem_u32(bars), empty0 = full0 + 8 * S, accf0 = full0 + 16 * S, acce0 = accf0 + 8 * NSLOT,
                 done = acce0 + 8 * NSLOT, ready = done + 8;

  pdl_trigger();
  if (warp == kProdWarp && lane == 0) {
    prefetch_tmap(&tmA);
    prefetch_tmap(&tmB);
    prefetch_tmap(&tmY);
  }
  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8 * s, 1);
      mbar_init(empty0 + 8 * s, 1);
    }
    for (int b = 0; b < NSLOT; ++b) {
      mbar_init(accf0 + 8 * b, 1);
      mbar_init(acce0 + 8 * b, 2 * 32 * kEpiWarps);  // both CTAs' epilogue threads
    }
    mbar_init(done, 1);
    mbar_init(ready, 1);
    s_fail = 0u;
    fence_mbar_init();
  }
  if (warp == kMmaWarp) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;\n" ::"r"(smem_u32(&tmem_slot)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;\n" ::: "memory");
  }
  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // both CTAs' barriers exist before either signals the other
  tc_fence_after();
  const uint32_t tmem = tmem_slot;
  const uint32_t full_lead = map_to_rank(full0, 0), acce_lead = map_to_rank(acce0, 0);
  pdl_wait();

  if (warp == kProdWarp) {
    // ---------------------------------------------------------------------- TMA producers (both CTAs)
    if (lane == 0) {
      bool ok = true;
      int g = 0;
      for (int t = pair; t < tiles && ok; t += npairs) {
        const int n0 = (t % NT) * BN, m0 = (t / NT) * 2 * kBM;
        for (int kb = 0; kb < nkb; ++kb, ++g) {
          const int s = g % S;
          if (!mbar_wait_bounded(empty0 + 8 * s, (uint32_t)(((g / S) & 1) ^ 1), kWaitBudgetCycles)) {
            ok = false;
            break;
          }
          if (rank == 0) mbar_arrive_expect_tx(full0 + 8 * s, 2 * (kABytes + GG::BHalf));
          tma_load_2d_pair(sA + (uint32_t)s * kABytes, &tmA, kb * BKe, m0 + kBM * (int)rank, full_lead + 8 * s);
          tma_load_2d_pair(sB + (uint32_t)s * GG::BHalf, &tmB, kb * BKe, n0 + (BN / 2) * (int)rank, full_lead + 8 * s);
        }
      }
      if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
      // the last stages are consumed (so their copies have landed) before this CTA can exit
      for (int j = g > S ? g - S : 0; j < g; ++j) {
        if (!mbar_wait_bounded(empty0 + 8 * (j % S), (uint32_t)((j / S) & 1), kWaitBudgetCycles)) {
          atomicOr(a.err, DEVERR_DRAIN_WAIT);
          break;
        }
      }
    }
  } else if (warp == kMmaWarp) {
    // ---------------------------------------------------------------------- MMA issuer (CTA 0)
    if (lane == 0 && rank == 0) {
      constexpr uint32_t idesc = idesc_f16(kMode == kModeBf16 ? 1u : 0u, BN, 2 * kBM);
      bool ok = true, known = false;  // known: this CTA's exactness scan has been read
      uint32_t fail = 0u;
      int g = 0, q = 0;
      // As in the single-CTA kernel: a W8A8 tile restarts in the next slot at each fold boundary
      // unless its row tile passed the exactness bound.
      for (int t = pair; t < tiles && ok; t += npairs) {
        int slot = q % NSLOT, kb0 = 0, next_fold = kb_per_chunk;
        if (q >= NSLOT &&
            !mbar_wait_bounded(acce0 + 8 * slot, (uint32_t)(((q / NSLOT) - 1) & 1), kWaitBudgetCycles)) {
          ok = false;
          break;
        }
        tc_fence_after();
        uint32_t d = tmem + (uint32_t)(slot * SC);
        for (int kb = 0; kb < nkb; ++kb, ++g) {
          if (kInt8 && kb == next_fold) {  // a fold boundary
            next_fold += kb_per_chunk;
            if (scan && !known) {
              if (!mbar_wait_bounded(ready, 0u, kWaitBudgetCycles)) {
                ok = false;
                break;
              }
              fail = s_fail;
              known = true;
            }
            if (!(scan && row_tile_exact(fail, t / NT))) {
              tc2_commit_both(accf0 + 8 * slot);
              ++q;
              slot = q % NSLOT;
              if (q >= NSLOT &&
                  !mbar_wait_bounded(acce0 + 8 * slot, (uint32_t)(((q / NSLOT) - 1) & 1), kWaitBudgetCycles)) {
                ok = false;
                break;
              }
              tc_fence_after();
              d = tmem + (uint32_t)(slot * SC);
              kb0 = kb;
            }
          }
          const int s = g % S;
          if (!mbar_wait_bounded(full0 + 8 * s, (uint32_t)((g / S) & 1), kWaitBudgetCycles)) {
            ok = false;
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int k16 = 0; k16 < kSwz / 32; ++k16) {  // 32 bytes of k per instruction
            const uint64_t ad = sdesc_swz(sA + (uint32_t)s * kABytes + 32u * k16);
            const uint64_t bd = sdesc_swz(sB + (uint32_t)s * GG::BHalf + 32u * k16);
            tc2_mma_m<kMode>(d, ad, bd, idesc, (kb == kb0 && k16 == 0) ? 0u : 1u);
          }
          tc2_commit_both(empty0 + 8 * s);
        }
        if (ok) tc2_commit_both(accf0 + 8 * slot);
        ++q;
      }
      if (!ok) atomicOr(a.err, DEVERR_PRODUCER_WAIT);
      tc2_commit(done);
      if (!mbar_wait_bounded(done, 0u, kWaitBudgetCycles)) atomicOr(a.err, DEVERR_DRAIN_WAIT);
    }
  } else {
    // ---------------------------------------------------------------------- epilogue warps 0-15 (both CTAs)
    if (scan) scan_exact(a, 2 * kBM, &s_fail, ready);
    const int quad = warp & 3, part = warp >> 2;
    const uint32_t lane_base = tmem + ((uint32_t)(32 * quad) << 16);
    const bool want_top = a.kind == EPI_F32 && a.top1 != nullptr;
    const uint32_t buf = stg + (uint32_t)(warp * kStageBufBytes);
    bool ok = true;
    int q = 0;
    for (int t = pair; t < tiles && ok; t += npairs) {
      const int n0 = (t % NT) * BN, m0 = (t / NT) * 2 * kBM;
      const int row = m0 + kBM * (int)rank + 32 * quad + lane;
      unsigned long long best = 0ull;
      auto emit = [&](int c0, const float (&v)[32]) {
        stage_cols32(a, &tmY, buf, m0 + kBM * (int)rank + 32 * quad, n0 + c0, lane, v, want_top, best);
      };
      if constexpr (kInt8) {
        constexpr int NG = (BN / 32 + kParts - 1) / kParts;  // this warp's 32-column groups: part + kParts i
        int isum[32 * NG];
#pragma unroll
        for (int j = 0; j < 32 * NG; ++j) isum[j] = 0;
        ColVals<NG> cv;  // before the first wait: the loads overlap the MMAs
        load_colvals<NG>(a, true, n0, part, BN, lane, cv);
        const float sx = row < a.M ? a.s_x[row] : 0.0f;
        const int nch = tile_chunks(t);
        if (nch == 1) {  // one exact fp32 accumulator: it is the INT32 sum as a float; dequantise directly
          const int slot = q % NSLOT;
          if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
            ok = false;
            atomicOr(a.err, DEVERR_CONSUMER_WAIT);
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int i = 0; i < NG; ++i) {
            const int g = part + kParts * i;
            if (g >= BN / 32) break;
            uint32_t r[32];
            tmem_ld32(lane_base + (uint32_t)(slot * SC + 32 * g), r);
            if (a.acc_dbg && row < a.M) {
#pragma unroll
              for (int j = 0; j < 32; ++j)
                if (n0 + 32 * g + j < a.N)
                  a.acc_dbg[(size_t)row * a.N + n0 + 32 * g + j] = __float2int_rn(__uint_as_float(r[j]));
            }
            float v[32];
            dequant32(a.bias != nullptr, sx, cv.sw[i], cv.b[i], r, v);
            emit(32 * g, v);
          }
          tc_fence_before();
          mbar_arrive_cluster(acce_lead + 8 * slot);
          ++q;
          if (want_top && row < a.M && best != 0ull) atomicMax(a.top_keys + row, best);
          continue;
        }
        for (int c = 0; c < nch; ++c, ++q) {
          const int slot = q % NSLOT;
          if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
            ok = false;
            atomicOr(a.err, DEVERR_CONSUMER_WAIT);
            break;
          }
          tc_fence_after();
#pragma unroll
          for (int i = 0; i < NG; ++i) {
            const int g = part + kParts * i;
            if (g >= BN / 32) break;
            uint32_t r[32];
            tmem_ld32(lane_base + (uint32_t)(slot * SC + 32 * g), r);
#pragma unroll
            for (int j = 0; j < 32; ++j) isum[32 * i + j] += __float2int_rn(__uint_as_float(r[j]));
          }
          tc_fence_before();
          mbar_arrive_cluster(acce_lead + 8 * slot);
        }
        if (!ok) break;
#pragma unroll
        for (int i = 0; i < NG; ++i) {
          const int g = part + kParts * i;
          if (g >= BN / 32) break;
          if (a.acc_dbg && row < a.M) {
#pragma unroll
            for (int j = 0; j < 32; ++j)
              if (n0 + 32 * g + j < a.N) a.acc_dbg[(size_t)row * a.N + n0 + 32 * g + j] = isum[32 * i + j];
          }
          float v[32];
          dequant32(a.bias != nullptr, sx, cv.sw[i], cv.b[i], &isum[32 * i], v);
          emit(32 * g, v);
        }
      } else {
        constexpr int NG = (BN / 32 + kParts - 1) / kParts;
        ColVals<NG> cv;  // before the wait: the loads overlap the MMAs
        load_colvals<NG>(a, kFp8, n0, part, BN, lane, cv);
        const float sx = kFp8 && row < a.M ? a.s_x[row] : 0.0f;
        const int slot = q % NSLOT;
        if (!mbar_wait_bounded(accf0 + 8 * slot, (uint32_t)((q / NSLOT) & 1), kWaitBudgetCycles)) {
          ok = false;
          atomicOr(a.err, DEVERR_CONSUMER_WAIT);
          break;
        }
        tc_fence_after();
#pragma unroll
        for (int i = 0; i < NG; ++i) {
          const int g = part + kParts * i;
          if (g >= BN / 32) break;
          uint32_t r[32];
          tmem_ld32(lane_base + (uint32_t)(slot * SC + 32 * g), r);
          float v[32];
          if constexpr (kFp8) {
            dequant32(a.bias != nullptr, sx, cv.sw[i], cv.b[i], r, v);
          } else {
#pragma unroll
            for (int j = 0; j < 32; ++j) v[j] = __uint_as_float(r[j]);
            if (a.bias) add_bias32(cv.b[i], v);
          }
          emit(32 * g, v);
        }
        tc_fence_before();
        mbar_arrive_cluster(acce_lead + 8 * slot);
        ++q;
      }
      if (want_top && row < a.M && best != 0ull) atomicMax(a.top_keys + row, best);
    }
    if (lane == 0) bulk_wait_all();  // this warp's output stores have completed
    __syncwarp();
    if (want_top) {
      __threadfence();
      named_bar_sync(1, 32 * kEpiWarps);
      if (threadIdx.x == 0) {
        const unsigned int prev = atomicAdd(a.grid_counter, 1u);
        s_flag = prev == gridDim.x - 1;
        if (s_flag) *a.grid_counter = 0u;
      }
      named_bar_sync(1, 32 * kEpiWarps);
      if (s_flag) {
        __threadfence();
        for (int t = threadIdx.x; t < a.M; t += 32 * kEpiWarps) {
          const unsigned long long key = atomicExch(a.top_keys + t, 0ull);
          a.top1[t] = (int32_t)(0xFFFFFFFFu - (uint32_t)(key & 0xFFFFFFFFull));
        }
      }
    }
    tc_fence_before();
  }
  __syncthreads();
  cluster_sync_all();  // neither CTA leaves while the other may still signal its barriers
  if (warp == kMmaWarp) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;\n" ::"r"(tmem), "r"(kTmemCols) : "memory");
  }
}

// The output's tensor map for the epilogue's TMA stores: 32 rows x 32 bf16 columns, or 16 (GeGLU
// output, fp32 logits), swizzled over the staged row's width.
w8a8_status make_out_map(const TcArgs& a, CUtensorMap* ty, const CUtensorMap& unused) {
  if (a.kind == EPI_BF16) return make_tmap_2d(ty, a.y, 2, (uint64_t)a.N, (uint64_t)a.M, (uint64_t)a.N * 2, 32, 32, 64);
  if (a.kind == EPI_GEGLU)
    return make_tmap_2d(ty, a.y, 2, (uint64_t)(a.N / 2), (uint64_t)a.M, (uint64_t)a.N, 16, 32, 32);
  if (a.logits) return make_tmap_2d(ty, a.logits, 4, (uint64_t)a.N, (uint64_t)a.M, (uint64_t)a.N * 4, 16, 32, 64);
  *ty = unused;  // top-1 only: nothing is stored
  return W8A8_OK;
}

template <int kMode, int kBN>
w8a8_status launch_t(const TcArgs& a, cudaStream_t st) {
  using GG = TcGeo<kMode, kBN>;
  constexpr int EB = elem_bytes(kMode), BKe = bk_elems(kMode);
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(gemm_tc_kernel<kMode, kBN>, cudaFuncAttributeMaxDynamicSharedMemorySize, GG::Smem));
    attr_set[dev] = true;
  }
  CUtensorMap ta, tb;
  W8A8_TRY(make_tmap_2d(&ta, a.A, EB, (uint64_t)a.K, (uint64_t)a.M, (uint64_t)a.K * EB, BKe,
                        (uint32_t)a_box_rows(a.M), kSwz));
  W8A8_TRY(make_tmap_2d(&tb, a.B, EB, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K * EB, BKe, GG::BN, kSwz));
  CUtensorMap ty;
  W8A8_TRY(make_out_map(a, &ty, ta));
  const long long tiles = (long long)((a.N + GG::BN - 1) / GG::BN) * ((a.M + kBM - 1) / kBM);
  const dim3 grid((unsigned)std::min<long long>(tiles * std::max(a.ksplit, 1), device_sms()));
  W8A8_CUDA(launch_pdl(gemm_tc_kernel<kMode, kBN>, grid, dim3(kThreads), (size_t)GG::Smem, st, ta, tb, ty, a));
  return W8A8_OK;
}

template <int kMode, int kBN>
w8a8_status launch_t2(const TcArgs& a, cudaStream_t st) {
  using GG = Tc2Geo<kMode, kBN>;
  constexpr int EB = elem_bytes(kMode), BKe = bk_elems(kMode);
  static bool attr_set[64] = {};
  int dev = 0;
  W8A8_CUDA(cudaGetDevice(&dev));
  if (dev >= 0 && dev < 64 && !attr_set[dev]) {
    W8A8_CUDA(cudaFuncSetAttribute(gemm_tc2_kernel<kMode, kBN>, cudaFuncAttributeMaxDynamicSharedMemorySize, GG::Smem));
    attr_set[dev] = true;
  }
  CUtensorMap ta, tb;
  W8A8_TRY(make_tmap_2d(&ta, a.A, EB, (uint64_t)a.K, (uint64_t)a.M, (uint64_t)a.K * EB, BKe, kBM, kSwz));
  W8A8_TRY(make_tmap_2d(&tb, a.B, EB, (uint64_t)a.K, (uint64_t)a.N, (uint64_t)a.K * EB, BKe, GG::BN / 2, kSwz));
  CUtensorMap ty;
  W8A8_TRY(make_out_map(a, &ty, ta));
  const long long tiles = (long long)((a.N + GG::BN - 1) / GG::BN) * ((a.M + 2 * kBM - 1) / (2 * kBM));
  const long long pairs = std::min<long long>(tiles, device_sms() / 2);
  W8A8_CUDA(launch_pdl(gemm_tc2_kernel<kMode, kBN>, dim3((unsigned)(2 * pairs)), dim3(kThreads), (size_t)GG::Smem, st,
                       ta, tb, ty, a));
  return W8A8_OK;
}

// Tile choice: CTA pairs on 256 tokens x 256 or 192 channels, or single CTAs on 128 x 128 or
// 128 x 64.  A persistent grid's time is taken as waves x the time of one SM's share of a tile (128
// tokens x BN channels), that share costing BN x {1, 1.32, 1.81, 2.7} for the four shapes (fitted
// to one-wave timings on K = 6912, where a narrower tile spends relatively more of each k step on
// operand traffic through shared memory; the last estimated from its operand bytes per MMA).
// Narrow tiles win where the wide ones would leave SMs idle, as at decode-sized token counts.
//
// Split-K: where a single-CTA bf16-output shape leaves more than half of the SMs without a tile
// (few tokens and a narrow output, as the attention projections and the down projection at decode
// batch sizes), the k range of every tile is cut into parts on different CTAs (at most one unit per
// SM, at least kMinKbPerPart stages per part).  Each CTA streams its part of the weights at the
// per-SM copy rate, so the spread is what reaches HBM bandwidth.
constexpr int kMinKbPerPart = 2;

// The parts are also capped at K / (4 R), so that the partials a tile's last unit reads back (KS R
// BN fp32) stay below half of the tile's weight bytes (BN K bf16), and fewer than kMinParts parts
// are not worth the arrival protocol.  Measured: 6-8 parts on q/k/v and o at 32 tokens save 1.5 us
// of 10-11, the down projection drops from 34 to 12-16 us, and q/k/v and o at 128 tokens (2 parts
// under the cap) would lose.
constexpr int kMinParts = 4;

// k parts of a single-CTA call on BN-column tiles (1: no split); split_ok: the caller gave the
// partials and tile counters the split needs
int split_parts(int mode, int M, int N, int K, int kind, bool split_ok, int bn, int sms) {
  const int nkb = (K + bk_elems(mode) - 1) / bk_elems(mode);
  const long long tiles = (long long)((N + bn - 1) / bn) * ((M + kBM - 1) / kBM);
  if (kind == EPI_BF16 && split_ok && 2 * tiles <= sms) {
    const int ks = std::min({(int)(sms / tiles), nkb / kMinKbPerPart, K / (4 * a_box_rows(M))});
    if (ks >= kMinParts) return ks;
  }
  return 1;
}

}  // namespace

TcChoice tc_choose(int mode, int M, int N, int K, int kind, bool split_ok, int sms) {
  const long long pairs = sms / 2;
  // ks k parts: ks units per tile, each with 1/ks of the k range, plus the partials' round trip
  // (taken as a third of a unit's time).  Counted from 256 tokens on the bf16 and W8A8 paths only:
  // there it picks split 128-column tiles over one wave of 64-column tiles (512 x 6912 -> 1152:
  // bf16 38.6 -> 32.4 us, W8A8 42.6 -> 33.4 us), while below it, and on the FP8 path, it measured
  // slower than the split-free model (128-token prefill 1.87 -> 2.22 ms; FP8 at 512 tokens 23 -> 29 us)
  const bool split_cost = M >= 256 && mode != kModeFp8;
  auto cost = [&](int bm, int bn, double unit, long long slots, int ks = 1) {
    const long long t = (long long)((N + bn - 1) / bn) * ((M + bm - 1) / bm) * ks;
    return (double)((t + slots - 1) / slots) * bn * unit / ks * (ks > 1 ? 1.33 : 1.0);
  };
  const double c256 = cost(2 * kBM, 256, 1.0, pairs), c192 = cost(2 * kBM, 192, 1.32, pairs),
               c128 = cost(kBM, 128, 1.81, 2 * pairs, split_cost ? split_parts(mode, M, N, K, kind, split_ok, 128, sms) : 1),
               c64 = cost(kBM, 64, 2.7, 2 * pairs, split_cost ? split_parts(mode, M, N, K, kind, split_ok, 64, sms) : 1);
  // W8A8 only: pairs on 256 x 128 tiles where the output is narrow but the single-CTA tiles would
  // not be split over k (they fill more than half of the SMs); four 128-column accumulator slots
  // keep the fold chunks of a long k range in flight (measured on 2048 x 6912 -> 1152: 42.7 us
  // against 45.7 us on single CTAs; the bf16 and FP8 paths measured no gain)
  const double p128 = mode == kModeI8 ? cost(2 * kBM, 128, 1.32, pairs) : 1e30;
  if (c256 <= c192 && c256 <= c128 && c256 <= c64 && c256 <= p128) return TcChoice{1, 256, 1};
  if (c192 <= c128 && c192 <= c64 && c192 <= p128) return TcChoice{1, 192, 1};
  const long long t128 = (long long)((N + 127) / 128) * ((M + kBM - 1) / kBM);
  if (mode == kModeI8 && 2 * t128 > sms && p128 < c128 && p128 < c64) return TcChoice{1, 128, 1};
  if (c128 <= c64) return TcChoice{0, 128, split_parts(mode, M, N, K, kind, split_ok, 128, sms)};
  return TcChoice{0, 64, split_parts(mode, M, N, K, kind, split_ok, 64, sms)};  // few tokens: spread the weights
}

namespace {

template <int kMode>
w8a8_status dispatch(TcArgs a, cudaStream_t st) {
  const TcChoice c = tc_choose(kMode, a.M, a.N, a.K, a.kind, a.partials && a.tile_counters, device_sms());
  a.ksplit = c.ksplit;
  if (c.pair) {
    if (c.bn == 256) return launch_t2<kMode, 256>(a, st);
    if (c.bn == 192) return launch_t2<kMode, 192>(a, st);
    return launch_t2<kMode, 128>(a, st);
  }
  if (c.bn == 128) return launch_t<kMode, 128>(a, st);
  return launch_t<kMode, 64>(a, st);
}

}  // namespace

bool tc_gemm_supported(int M, int N, int K, int kind, bool want_top, int max_top) {
  if (M < 1 || N < 16 || K < 16 || K % 16 != 0 || N % 16 != 0) return false;
  if (kind != EPI_BF16 && kind != EPI_GEGLU && kind != EPI_F32) return false;
  if (want_top && M > max_top) return false;
  return true;
}

size_t tc_split_partial_bytes(int M, int sms) {
  // at most one unit per SM, BN <= 128 on the single-CTA kernel, R = a_box_rows(M) rows per unit
  return (size_t)std::max(sms, 1) * 128 * (size_t)a_box_rows(std::max(M, 1)) * 4;
}

w8a8_status launch_tc_gemm(int mode, const TcArgs& a, cudaStream_t st) {
  if (a.M == 0 || a.N == 0) return W8A8_OK;
  void *v0, *v1;
  take_kernel_events(&v0, &v1);
  cudaEvent_t e0 = reinterpret_cast<cudaEvent_t>(v0), e1 = reinterpret_cast<cudaEvent_t>(v1);
  if (e0) W8A8_CUDA(cudaEventRecord(e0, st));
  const w8a8_status s = mode == TC_FP8 ? dispatch<kModeFp8>(a, st)
                        : mode == TC_I8 ? dispatch<kModeI8>(a, st)
                                        : dispatch<kModeBf16>(a, st);
  if (e1) W8A8_CUDA(cudaEventRecord(e1, st));
  return s;
}

}  // namespace w8a8
