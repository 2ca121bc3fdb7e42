// common.cuh -- shared host/device plumbing of libssm: status codes, the
// device error word, the wait limit and argument-check helpers.
#pragma once

#include <cuda_runtime.h>
#include <cstdint>

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

inline ssm_status launch_status() {
  cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SSM_OK : SSM_ERR_CUDA;
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

}  // namespace ssm
