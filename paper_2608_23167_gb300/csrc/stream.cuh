// stream.cuh -- the vocabulary-streaming plumbing shared by the unmasking pass
// and the suffix top-k pass: rows of logits cut into segments (work items dealt
// round-robin to persistent CTAs), each thread copying its own 16-byte slices
// of successive chunks into a private shared-memory ring with cp.async.
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

// Walks the chunks of this CTA's work items (masked rows only) in order.
struct ChunkIter {
  int64_t item, off, bytes, e0, row;
  bool valid;
};

template <typename T>
__device__ __forceinline__ void chunk_seek(ChunkIter& it, int64_t vocab, int64_t seg_elems, int n_seg,
                                           int64_t n_items, const uint8_t* __restrict__ masked) {
  // advance to the next item that has a masked row (every row when masked is null),
  // if the current one is exhausted
  while (it.item < n_items && (it.off >= it.bytes)) {
    it.item += gridDim.x;
    it.off = 0;
    if (it.item >= n_items) break;
    it.row = it.item / n_seg;
    if (masked && !masked[it.row]) {
      it.bytes = 0;
      continue;
    }
    it.e0 = (it.item - it.row * n_seg) * seg_elems;
    it.bytes = (min(vocab, it.e0 + seg_elems) - it.e0) * static_cast<int64_t>(sizeof(T));
  }
  it.valid = it.item < n_items;
}

}  // namespace ssm
