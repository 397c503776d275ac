// Host helper: 2-D TMA tensor maps (cuTensorMapEncodeTiled reached through the runtime's driver
// entry-point query, so the library does not link libcuda).
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace w8a8 {

// Row-major [rows, inner] tensor of `elem_bytes`-byte (1, 2 or 4) elements with a row pitch of `pitch_bytes`;
// the box is [box_rows, box_inner], zero-filled outside the tensor, with a 128-, 64- or 32-byte
// swizzle (box_inner * elem_bytes at most that many bytes) or none (swizzle_bytes 0: rows of the box
// packed one after another).
w8a8_status make_tmap_2d(CUtensorMap* map, const void* base, int elem_bytes, uint64_t inner, uint64_t rows,
                         uint64_t pitch_bytes, uint32_t box_inner, uint32_t box_rows, int swizzle_bytes = 128);

}  // namespace w8a8
