// cache.cu -- prefix-cache append at a block boundary (the prefix-caching
// setting "+PC." of Sec. 4.8, Table 4): once a block is decoded, the keys and
// values of its rows enter the cache that later steps read (keys rotated at the
// rows' positions, as every cached key is; Sec. 3.2 "Sparse Input
// Construction": tokens keep their original positions).
//
// cache_append_kernel: persistent warps, one (sequence, row) at a time.  The
// row's D/2 angles are formed once (two per lane) and shared through shared
// memory; a lane then owns eight rotation pairs of one head vector (D/16 lanes
// per head, 16-byte accesses, two head passes in flight).  The rotation is
// rope.cuh's, so a key appended here carries the same bf16 bits as the same key
// rotated by the attention's pre-pass.  Values are copied.
#include <cuda_bf16.h>

#include <algorithm>

#include "common.cuh"
#include "rope.cuh"

namespace ssm {
namespace {

constexpr int kAppendWarps = 8;

template <int D>
__global__ void __launch_bounds__(kAppendWarps * 32) cache_append_kernel(
    const __nv_bfloat16* __restrict__ k_new, const __nv_bfloat16* __restrict__ v_new,
    const int32_t* __restrict__ pos, int32_t batch, int32_t n_rows, int32_t h_kv, const RopeFreqs<D> freqs,
    __nv_bfloat16* __restrict__ k_cache, __nv_bfloat16* __restrict__ v_cache, int64_t cache_rows,
    int64_t start_row) {
  pdl_enter();
  constexpr int LPH = D / 16;    // lanes per head vector: eight rotation pairs per lane
  constexpr int HPP = 32 / LPH;  // head vectors per warp pass
  __shared__ uint64_t turn[D / 2];
  __shared__ float s_cs[kAppendWarps][D / 2], s_sn[kAppendWarps][D / 2];
  if (threadIdx.x < D / 2) turn[threadIdx.x] = freqs.turn[threadIdx.x];
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int sub = lane % LPH, hoff = lane / LPH;
  const int64_t total = static_cast<int64_t>(batch) * n_rows;
  // persistent warps over (sequence, row): the CTA's table is made once
  for (int64_t r = static_cast<int64_t>(blockIdx.x) * kAppendWarps + warp; r < total;
       r += static_cast<int64_t>(gridDim.x) * kAppendWarps) {
    const int64_t b = r / n_rows;
    const int i = static_cast<int>(r - b * n_rows);
    // each pair's angle once per row (a lane takes pairs lane, lane + 32), shared through shared memory
    const int32_t ps = pos[i];
    __syncwarp();
#pragma unroll
    for (int t = lane; t < D / 2; t += 32) rope_sincos(ps, turn[t], s_sn[warp][t], s_cs[warp][t]);
    __syncwarp();
    float cs0[4], cs1[4], sn0[4], sn1[4];
#pragma unroll
    for (int t = 0; t < 4; ++t) {
      cs0[t] = s_cs[warp][8 * sub + t];
      cs1[t] = s_cs[warp][8 * sub + 4 + t];
      sn0[t] = s_sn[warp][8 * sub + t];
      sn1[t] = s_sn[warp][8 * sub + 4 + t];
    }
    const int64_t src_row = r;
    const int64_t dst_row = b * cache_rows + start_row + i;
    // two head passes per iteration: eight 16-byte loads in flight per lane
    for (int h0 = hoff; h0 < h_kv; h0 += 2 * HPP) {
      uint4 x1[2], x2[2], v1[2], v2[2];
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int h = h0 + u * HPP;
        if (h < h_kv) {
          const __nv_bfloat16* ks = k_new + (src_row * h_kv + h) * D + 8 * sub;
          const __nv_bfloat16* vs = v_new + (src_row * h_kv + h) * D + 8 * sub;
          x1[u] = *reinterpret_cast<const uint4*>(ks);
          x2[u] = *reinterpret_cast<const uint4*>(ks + D / 2);
          v1[u] = *reinterpret_cast<const uint4*>(vs);
          v2[u] = *reinterpret_cast<const uint4*>(vs + D / 2);
        }
      }
#pragma unroll
      for (int u = 0; u < 2; ++u) {
        const int h = h0 + u * HPP;
        if (h >= h_kv) continue;
        uint2 ya, yb, yc, yd;
        rope_rotate4(make_uint2(x1[u].x, x1[u].y), make_uint2(x2[u].x, x2[u].y), cs0, sn0, ya, yb);
        rope_rotate4(make_uint2(x1[u].z, x1[u].w), make_uint2(x2[u].z, x2[u].w), cs1, sn1, yc, yd);
        __nv_bfloat16* kd = k_cache + (dst_row * h_kv + h) * D + 8 * sub;
        __nv_bfloat16* vd = v_cache + (dst_row * h_kv + h) * D + 8 * sub;
        *reinterpret_cast<uint4*>(kd) = make_uint4(ya.x, ya.y, yc.x, yc.y);
        *reinterpret_cast<uint4*>(kd + D / 2) = make_uint4(yb.x, yb.y, yd.x, yd.y);
        *reinterpret_cast<uint4*>(vd) = v1[u];
        *reinterpret_cast<uint4*>(vd + D / 2) = v2[u];
      }
    }
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
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int64_t warps_needed = (static_cast<int64_t>(batch) * n_rows + ssm::kAppendWarps - 1) / ssm::kAppendWarps;
  const int grid = static_cast<int>(std::min<int64_t>(warps_needed, 8ll * ssm::num_sms()));
  const auto* kn = static_cast<const __nv_bfloat16*>(k_new);
  const auto* vn = static_cast<const __nv_bfloat16*>(v_new);
  auto* kc = static_cast<__nv_bfloat16*>(k_cache);
  auto* vc = static_cast<__nv_bfloat16*>(v_cache);
  if (head_dim == 128)
    ssm::launch_k(ssm::cache_append_kernel<128>, dim3(grid), dim3(ssm::kAppendWarps * 32), 0, st, kn, vn, pos,
                  batch, n_rows, h_kv, ssm::rope_freqs<128>(rope_theta), kc, vc, cache_rows, start_row);
  else
    ssm::launch_k(ssm::cache_append_kernel<64>, dim3(grid), dim3(ssm::kAppendWarps * 32), 0, st, kn, vn, pos,
                  batch, n_rows, h_kv, ssm::rope_freqs<64>(rope_theta), kc, vc, cache_rows, start_row);
  return ssm::launch_status();
}

}  // extern "C"
