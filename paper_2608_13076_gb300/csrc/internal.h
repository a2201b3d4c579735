// internal.h -- host-side helpers shared by the entry points (not part of the ABI).
#pragma once
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>

#include "../../include/spade.h"

namespace spade {

// Records a thread-local message for spade_last_error() and returns `s`.
spade_status fail(spade_status s, const char *fmt, ...);
// Maps a CUDA runtime error to SPADE_ERR_CUDA with a message naming `what`.
spade_status cuda_fail(cudaError_t e, const char *what);

// Checks that the current device is sm_103 and returns its SM count.
spade_status device_info(int *num_sms, int *device);

// Encodes a 2-D bf16 tensor map [rows, inner] with row stride
// `row_stride_bytes`, box {box_inner, box_rows}, 128-byte swizzle, zero fill
// out of bounds.  Returns false (with a message recorded) on failure.
bool encode_tmap_bf16_sw128(CUtensorMap *map, const void *base, uint64_t inner, uint64_t rows,
                            uint64_t row_stride_bytes, uint32_t box_inner, uint32_t box_rows);

// Encodes a 3-D view of a row-major bf16 matrix [rows, cols] (cols a multiple
// of 64): dims {64, rows, cols/64}, strides {cols*2, 128} bytes, box
// {64, box_rows, box_slabs}, 128-byte swizzle.  One box fetches box_rows rows
// and lands them as box_slabs slabs of [box_rows][64], back to back; box_slabs
// = 0 means all cols/64 slabs (whole rows).
bool encode_tmap_rows_by_slab(CUtensorMap *map, const void *base, uint64_t rows, uint32_t cols,
                              uint32_t box_rows, uint32_t box_slabs = 0);

inline bool aligned(const void *p, uintptr_t a) {
  return (reinterpret_cast<uintptr_t>(p) % a) == 0;
}
inline size_t round_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace spade
