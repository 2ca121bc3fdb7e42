// common.cuh -- shared host/device plumbing of libssm: status codes, the
// device error word, the wait limit and argument-check helpers.
#pragma once

#include <cuda_runtime.h>
#include <cstdint>
#include <utility>

#include "ssm.h"

namespace ssm {

// Records the first device-side error of any libssm kernel (0 = none).
__device__ __forceinline__ void record_error(unsigned* err, unsigned code) {
  if (err) atomicCAS(err, 0u, code);
}

// Device address of the error word for the current device (created on first use).
unsigned* device_error_word();

// Current wait limit for bounded device-side spins, in nanoseconds.
uint64_t wait_limit_ns();

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

inline int num_sms() {
  int dev = 0, n = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return 148;
  if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 148;
  return n;
}

// CTAs of `kernel` that fit on one SM at `threads` threads and `smem` bytes of dynamic shared
// memory (at least 1): the grid size of a persistent kernel is this times the SM count.
template <typename Kernel>
inline int resident_ctas(Kernel kernel, int threads, size_t smem) {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kernel, threads, smem) != cudaSuccess || n < 1) return 1;
  return n;
}

inline ssm_status launch_status() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SSM_OK : SSM_ERR_CUDA;
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Programmatic dependent launch.  Every libssm kernel launched directly on a stream carries
// the programmatic stream serialization attribute and every kernel begins with pdl_enter():
// griddepcontrol.wait blocks
// until the grids it depends on have completed and their memory is visible (a kernel that
// follows a non-libssm kernel or a copy waits for it as usual), then launch_dependents lets
// the next kernel of the stream be scheduled while this one runs.  The next kernel's CTAs take
// SM resources only as they free up and block in their own wait, so a dependent kernel's
// launch latency and CTA start-up overlap this kernel's tail instead of following it.  Every
// thread executes the wait before touching memory and before any return, so a kernel can
// complete only after everything earlier on the stream has.
__device__ __forceinline__ void pdl_enter() {
  asm volatile("griddepcontrol.wait;" ::: "memory");
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

template <typename... KArgs, typename... Args>
inline void launch_k(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                     Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  // Direct launches only: replays of a captured CUDA graph already start each node right after
  // its predecessor, and measured slower with programmatic edges, so launches being captured
  // are ordinary ones (pdl_enter() is then a no-op wait)
  cudaStreamCaptureStatus cap = cudaStreamCaptureStatusNone;
  cudaStreamIsCapturing(st, &cap);
  cfg.numAttrs = cap == cudaStreamCaptureStatusNone ? 1 : 0;
  cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);  // errors: read by launch_status()
}

// launch_k with programmatic dependent launch also while the stream is being captured (a
// programmatic edge in the graph).  Used for the unmasking's commit kernel, whose few small CTAs
// start beside the stream kernel's; the same edge in front of the attention forward and of the
// unmasking's stream kernel made the graph-replayed step slower (the long sweep 503 -> 541 us).
template <typename... KArgs, typename... Args>
inline void launch_k_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                         Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  cudaLaunchKernelEx(&cfg, kernel, std::forward<Args>(args)...);  // errors: read by launch_status()
}

}  // namespace ssm
