// tcgen05 building blocks shared by the tensor-core GEMMs (inline PTX): tensor-memory fences, the
// shared-memory matrix descriptor of a 128-byte-swizzled K-major tile, the instruction descriptor,
// single-CTA MMA issue and commit, and the 32-column tensor-memory load.
#pragma once

#include "common.cuh"

namespace w8a8 {

constexpr int kTcSwz = 128;  // swizzle span in bytes of the operand tiles (TMA and the descriptors agree)

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;\n" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;\n" ::: "memory"); }

// Shared-memory matrix descriptor of a K-major tile swizzled over kTcSwz bytes: rows of kTcSwz bytes,
// 8-row groups 8 kTcSwz bytes apart (stride byte offset), descriptor version 1, layout SWIZZLE_128B
// (2) or SWIZZLE_64B (4).
__device__ __forceinline__ uint64_t sdesc_swz(uint32_t saddr) {
  uint64_t d = 0;
  d |= (uint64_t)((saddr & 0x3FFFFu) >> 4);
  d |= (uint64_t)1 << 16;                       // leading byte offset (unused by swizzled K-major layouts)
  d |= (uint64_t)((8 * kTcSwz) >> 4) << 32;       // stride byte offset
  d |= (uint64_t)1 << 46;                       // version
  d |= (uint64_t)(kTcSwz == 128 ? 2 : 4) << 61;   // layout
  return d;
}

// Instruction descriptor of kind::f16 / kind::f8f6f4: fp32 accumulator (bits 4-5 = 1), A and B
// format at bits 7-9 and 10-12 (kind::f16: fp16 0, bf16 1; kind::f8f6f4: e4m3 0), both K-major,
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
__device__ __forceinline__ void tc_mma_f8(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc,
                                          uint32_t accumulate) {
  asm volatile(
      "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
      " tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}\n" ::"r"(d_tmem),
      "l"(a_desc), "l"(b_desc), "r"(idesc), "r"(accumulate)
      : "memory");
}
__device__ __forceinline__ void tc_commit(uint32_t bar) {
  asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];\n" ::"r"(bar) : "memory");
}
// 32 consecutive accumulator columns of this thread's lane; the wait sits in the same statement, so
// no use of r can be scheduled before the load has completed.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t (&r)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, "
      "%15, %16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];\n"
      "tcgen05.wait::ld.sync.aligned;\n"
      : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
        "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
        "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
        "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
      : "r"(taddr)
      : "memory");
}


constexpr int kKbPerChunk = 1024 / (kTcSwz / 2);  // 64-k fp16 stages per exact fp32 chunk of 1024 k
// W8A8 chunk length in stages for a range of len stages: the fewest chunks of at most kKbPerChunk
// stages, of equal length (the last one shorter), so that the epilogue's fold of one chunk overlaps
// the MMAs of a chunk as long as itself rather than those of a short remainder (1152 k: 576 + 576,
// not 1024 + 128).
__host__ __device__ constexpr int chunk_stages(int len) {
  return len <= kKbPerChunk ? (len > 0 ? len : 1)
                            : (len + (len + kKbPerChunk - 1) / kKbPerChunk - 1) / ((len + kKbPerChunk - 1) / kKbPerChunk);
}
__host__ __device__ constexpr int chunk_count(int len) {
  return len <= 0 ? 1 : (len + chunk_stages(len) - 1) / chunk_stages(len);
}
// The fold exists because a fp32 sum of integer products is exact only while every partial sum
// stays within 2^24.  Weight codes are at most 127 in magnitude, so for token t every partial sum
// of its products, in any order or grouping, is bounded by 127 sum_k |q_tk|: a tile whose tokens
// all have sum_k |q_tk| <= kExactQsum needs no fold at all (one accumulator over the whole k
// range, exact, as the bf16 path runs).  The bound is data-dependent; the quantiser reports the
// sums, and tiles that fail it take the chunked path.
constexpr int kExactQsum = (1 << 24) / 127;  // 132104: 127 x 132104 <= 2^24

}  // namespace w8a8
