// eos.cu -- early termination after a decoded block (Sec. 3.2 "Early
// Termination": generation halts once an end-of-sequence token appears, checked
// after each decoding block).  For every sequence still running, if the block
// just decoded holds the EOS token, the sequence is marked finished and every
// generated position after its first EOS is filled with EOS, so later blocks
// have nothing left to decode.
//
// early_stop_kernel: one CTA per sequence; the threads find the block's first
// EOS with a shared-memory minimum, then fill the tail with strided stores.
#include "common.cuh"

namespace ssm {
namespace {

constexpr int kEosThreads = 256;

__global__ void __launch_bounds__(kEosThreads) early_stop_kernel(int32_t* __restrict__ tokens, int32_t gen_len,
                                                                 int32_t block_len, int32_t block_idx, int32_t eos_id,
                                                                 uint8_t* __restrict__ finished,
                                                                 int32_t* __restrict__ n_active) {
  pdl_enter();
  __shared__ int s_first;
  const int64_t seq = blockIdx.x;
  if (finished[seq]) return;   // uniform over the CTA
  if (threadIdx.x == 0) s_first = INT32_MAX;
  __syncthreads();
  int32_t* row = tokens + seq * gen_len;
  const int b0 = block_idx * block_len;
  for (int j = threadIdx.x; j < block_len; j += kEosThreads)
    if (row[b0 + j] == eos_id) atomicMin(&s_first, b0 + j);
  __syncthreads();
  const int first = s_first;
  if (first == INT32_MAX) {
    if (n_active && threadIdx.x == 0) atomicAdd(n_active, 1);
    return;
  }
  if (threadIdx.x == 0) finished[seq] = 1;
  for (int p = first + 1 + threadIdx.x; p < gen_len; p += kEosThreads) row[p] = eos_id;
}

}  // namespace
}  // namespace ssm

extern "C" ssm_status ssm_early_stop(int32_t* tokens, int32_t batch, int32_t gen_len, int32_t block_len,
                                     int32_t block_idx, int32_t eos_id, uint8_t* finished, int32_t* n_active,
                                     ssm_stream_t stream) {
  if (batch < 0 || gen_len <= 0 || block_len <= 0 || block_idx < 0) return SSM_ERR_INVALID_ARG;
  if (gen_len % block_len != 0) return SSM_ERR_SHAPE;
  if (static_cast<int64_t>(block_idx + 1) * block_len > gen_len) return SSM_ERR_INVALID_ARG;
  if (batch == 0) return SSM_OK;
  if (!tokens || !finished) return SSM_ERR_INVALID_ARG;
  if (batch > INT32_MAX / 2) return SSM_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (n_active && cudaMemsetAsync(n_active, 0, sizeof(int32_t), st) != cudaSuccess) return SSM_ERR_CUDA;
  ssm::launch_k(ssm::early_stop_kernel, dim3(batch), dim3(ssm::kEosThreads), 0, st,
           tokens, gen_len, block_len, block_idx, eos_id,
                                                             finished, n_active);
  return ssm::launch_status();
}
