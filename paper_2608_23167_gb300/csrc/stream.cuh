// stream.cuh -- the vocabulary-streaming plumbing of the unmasking pass (and the
// bf16 helpers the suffix top-k pass shares): rows of logits cut into 16 KB
// stages, each CTA walking one contiguous range of them, each thread copying its
// own 16-byte slices of successive stages into a private shared-memory ring with
// cp.async.
#pragma once

#include <cuda_bf16.h>

#include <cstdint>

#include "sm100_ptx.cuh"

namespace ssm {

__device__ __forceinline__ float lo_bf16(uint32_t w) { return __uint_as_float(w << 16); }
__device__ __forceinline__ float hi_bf16(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

// 16-byte asynchronous global -> shared copy (L2 only, bypassing L1).
__device__ __forceinline__ void cp_async16(void* dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(dst)), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() {
  asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// A position in the streaming work: stage g of the masked rows' 16 KB stages,
// numbered row-major over the call (stage g = row * n_stage + j covers elements
// [j * stage_elems, min(vocab, (j + 1) * stage_elems)) of the row).  Each CTA
// walks one contiguous range of stages, so every CTA gets the same number of
// stages whatever the row length, and a range ends a row's fold only where it
// crosses a row boundary.  The cursor advances without divisions (one 64-bit
// division when a range starts) and reads a row's mask once, on entering it.
struct StageCursor {
  int64_t g;      // current stage (>= the range end once exhausted)
  int64_t row;    // its row
  int64_t e0;     // its first element
  int32_t j;      // its index within the row
  int32_t bytes;  // its length in bytes
};

// Skips whole unmasked rows (none when masked is null) from the cursor's stage on, then
// describes the stage it stops at (if it is below end).
template <typename T>
__device__ __forceinline__ void stage_settle(StageCursor& c, int64_t end, int32_t n_stage, int64_t stage_elems,
                                             int64_t vocab, const uint8_t* __restrict__ masked) {
  while (c.g < end && masked && !masked[c.row]) {
    c.g += n_stage - c.j;
    ++c.row;
    c.j = 0;
  }
  c.e0 = static_cast<int64_t>(c.j) * stage_elems;
  c.bytes = static_cast<int32_t>((min(vocab, c.e0 + stage_elems) - c.e0) * static_cast<int64_t>(sizeof(T)));
}

// Cursor at the first stage at or after g, below end, of a masked row.
template <typename T>
__device__ __forceinline__ StageCursor stage_begin(int64_t g, int64_t end, int32_t n_stage, int64_t stage_elems,
                                                   int64_t vocab, const uint8_t* __restrict__ masked) {
  StageCursor c;
  c.g = g;
  c.row = g / n_stage;
  c.j = static_cast<int32_t>(g - c.row * n_stage);
  stage_settle<T>(c, end, n_stage, stage_elems, vocab, masked);
  return c;
}

// The next stage of a masked row, below end.
template <typename T>
__device__ __forceinline__ void stage_next(StageCursor& c, int64_t end, int32_t n_stage, int64_t stage_elems,
                                           int64_t vocab, const uint8_t* __restrict__ masked) {
  ++c.g;
  if (++c.j == n_stage) {
    ++c.row;
    c.j = 0;
    stage_settle<T>(c, end, n_stage, stage_elems, vocab, masked);
  } else {
    c.e0 += stage_elems;
    c.bytes = static_cast<int32_t>((min(vocab, c.e0 + stage_elems) - c.e0) * static_cast<int64_t>(sizeof(T)));
  }
}

}  // namespace ssm
