// cache.cu -- prefix-cache append at a block boundary (the prefix-caching
// setting "+PC." of Sec. 4.8, Table 4): once a block is decoded, the keys and
// values of its rows enter the cache that later steps read (keys rotated at the
// rows' positions, as every cached key is; Sec. 3.2 "Sparse Input
// Construction": tokens keep their original positions).
//
// cache_append_kernel: one warp per (sequence, row).  A lane owns four
// rotation pairs of one head vector (D/8 lanes per head, 8-byte accesses), the
// rotation is rope.cuh's, so a key appended here carries the same bf16 bits as
// the same key rotated by the attention's pre-pass.  Values are copied.
#include <cuda_bf16.h>

#include "common.cuh"
#include "rope.cuh"

namespace ssm {
namespace {

constexpr int kAppendWarps = 8;

template <int D>
__global__ void __launch_bounds__(kAppendWarps * 32) cache_append_kernel(
    const __nv_bfloat16* __restrict__ k_new, const __nv_bfloat16* __restrict__ v_new,
    const int32_t* __restrict__ pos, int32_t n_rows, int32_t h_kv, float theta,
    __nv_bfloat16* __restrict__ k_cache, __nv_bfloat16* __restrict__ v_cache, int64_t cache_rows,
    int64_t start_row) {
  constexpr int LPH = D / 8;     // lanes per head vector
  constexpr int HPP = 32 / LPH;  // head vectors per warp pass
  __shared__ double inv_freq[D / 2];
  if (threadIdx.x < D / 2) inv_freq[threadIdx.x] = rope_inv_freq(theta, threadIdx.x, D);
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane % LPH, hoff = lane / LPH;
  const int64_t b = blockIdx.y;
  const int i = blockIdx.x * kAppendWarps + warp;
  if (i >= n_rows) return;
  float cs[4], sn[4];
#pragma unroll
  for (int t = 0; t < 4; ++t) rope_sincos(pos[i], inv_freq[4 * sub + t], sn[t], cs[t]);
  const int64_t src_row = b * n_rows + i;
  const int64_t dst_row = b * cache_rows + start_row + i;
  for (int h = hoff; h < h_kv; h += HPP) {
    const __nv_bfloat16* ks = k_new + (src_row * h_kv + h) * D;
    const __nv_bfloat16* vs = v_new + (src_row * h_kv + h) * D;
    __nv_bfloat16* kd = k_cache + (dst_row * h_kv + h) * D;
    __nv_bfloat16* vd = v_cache + (dst_row * h_kv + h) * D;
    const uint2 x1 = *reinterpret_cast<const uint2*>(ks + 4 * sub);
    const uint2 x2 = *reinterpret_cast<const uint2*>(ks + D / 2 + 4 * sub);
    const uint2 v1 = *reinterpret_cast<const uint2*>(vs + 4 * sub);
    const uint2 v2 = *reinterpret_cast<const uint2*>(vs + D / 2 + 4 * sub);
    uint2 y1, y2;
    rope_rotate4(x1, x2, cs, sn, y1, y2);
    *reinterpret_cast<uint2*>(kd + 4 * sub) = y1;
    *reinterpret_cast<uint2*>(kd + D / 2 + 4 * sub) = y2;
    *reinterpret_cast<uint2*>(vd + 4 * sub) = v1;
    *reinterpret_cast<uint2*>(vd + D / 2 + 4 * sub) = v2;
  }
}

}  // namespace
}  // namespace ssm

extern "C" {

ssm_status ssm_cache_append(const void* k_new, const void* v_new, const int32_t* pos, int32_t batch,
                            int32_t n_rows, int32_t h_kv, int32_t head_dim, float rope_theta, void* k_cache,
                            void* v_cache, int64_t cache_rows, int64_t start_row, ssm_stream_t stream) {
  if (batch < 0 || n_rows < 0 || h_kv <= 0 || cache_rows < 0 || start_row < 0) return SSM_ERR_INVALID_ARG;
  if (!(rope_theta >= 0.f)) return SSM_ERR_INVALID_ARG;
  if (head_dim != 64 && head_dim != 128) return SSM_ERR_UNSUPPORTED;
  if (start_row + static_cast<int64_t>(n_rows) > cache_rows) return SSM_ERR_CAPACITY;
  if (batch == 0 || n_rows == 0) return SSM_OK;
  if (!k_new || !v_new || !pos || !k_cache || !v_cache) return SSM_ERR_INVALID_ARG;
  if (!ssm::aligned16(k_new) || !ssm::aligned16(v_new) || !ssm::aligned16(k_cache) || !ssm::aligned16(v_cache))
    return SSM_ERR_INVALID_ARG;
  if (batch > 65535) return SSM_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const dim3 grid((n_rows + ssm::kAppendWarps - 1) / ssm::kAppendWarps, batch);
  const auto* kn = static_cast<const __nv_bfloat16*>(k_new);
  const auto* vn = static_cast<const __nv_bfloat16*>(v_new);
  auto* kc = static_cast<__nv_bfloat16*>(k_cache);
  auto* vc = static_cast<__nv_bfloat16*>(v_cache);
  if (head_dim == 128)
    ssm::cache_append_kernel<128><<<grid, ssm::kAppendWarps * 32, 0, st>>>(kn, vn, pos, n_rows, h_kv, rope_theta,
                                                                         kc, vc, cache_rows, start_row);
  else
    ssm::cache_append_kernel<64><<<grid, ssm::kAppendWarps * 32, 0, st>>>(kn, vn, pos, n_rows, h_kv, rope_theta,
                                                                        kc, vc, cache_rows, start_row);
  return ssm::launch_status();
}

}  // extern "C"
