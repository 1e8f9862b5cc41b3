// Tensor maps (TMA descriptors) over the [B][H][N][128] bf16 tensors.
#pragma once

#include <cuda.h>

#include "common.cuh"

namespace rola {

// The tensor viewed as 4-D (d within a 64-wide chunk, token, chunk, head): one
// 64 x rows x 2 x 1 box brings `rows` tokens (64: a whole block, 16 KB) in as
// [chunk][row][64], 128-byte swizzle; rows past N read as zero.
bool make_block_map(CUtensorMap* m, const void* ptr, const Shape& s, int rows = 64);

// The tensor viewed as 3-D (d, token, head) with 64 x 64 boxes: one d-chunk of
// a 64-token block, 8 KB, 128-byte swizzle; rows past N read as zero.
bool make_chunk_map(CUtensorMap* m, const void* ptr, const Shape& s);

}  // namespace rola
