// select.cu -- structured suffix selection (Sec. 3.2, Eqs. 1-5).
//
// Each thread classifies suffix positions independently (a closed-form
// membership test per position), and the CTA compacts the kept positions in
// ascending order with warp ballots and a block-wide prefix sum.  One CTA per
// selection; a batch of selections is one launch.
#include <algorithm>
#include <vector>

#include "common.cuh"
#include "suffix_geom.cuh"

namespace ssm {
namespace {

void host_counts(const ssm_suffix_cfg& c, int32_t* nl, int32_t* nmid, int32_t* nt) {
  region_counts(make_geom(c), *nl, *nmid, *nt);
}

ssm_status check_cfg(const ssm_suffix_cfg* c) {
  if (!c) return SSM_ERR_INVALID_ARG;
  if (c->block_len <= 0 || c->gen_len <= 0 || c->prompt_len < 0) return SSM_ERR_INVALID_ARG;
  if (c->gen_len % c->block_len != 0) return SSM_ERR_SHAPE;
  if (c->block_idx < 0 || c->block_idx >= c->gen_len / c->block_len) return SSM_ERR_INVALID_ARG;
  if (c->local_budget < 0 || c->middle_budget < 0 || c->tail_budget < 0) return SSM_ERR_INVALID_ARG;
  if (static_cast<int64_t>(c->prompt_len) + c->gen_len > INT32_MAX) return SSM_ERR_INVALID_ARG;
  return SSM_OK;
}

constexpr int kSelThreads = 256;
constexpr int kSelMaxPerLaunch = 64;  // keeps the kernel parameter block under 4 KB

struct SelectBatch {
  ssm_suffix_cfg cfg[kSelMaxPerLaunch];
  int64_t offset[kSelMaxPerLaunch];
};

__global__ void __launch_bounds__(kSelThreads) select_kernel(const __grid_constant__ SelectBatch batch,
                                                             int32_t* __restrict__ positions) {
  pdl_enter();
  __shared__ int32_t warp_tot[kSelThreads / 32];
  __shared__ int32_t base_s;
  const ssm_suffix_cfg cfg = batch.cfg[blockIdx.x];
  int32_t* out = positions + batch.offset[blockIdx.x];
  const SuffixGeom g = make_geom(cfg);
  if (g.n_sb <= 0) return;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (threadIdx.x == 0) base_s = 0;
  __syncthreads();
  for (int64_t start = g.s0; start < g.end; start += kSelThreads) {
    const int64_t pos = start + threadIdx.x;
    const bool k = pos < g.end && keeps(g, pos);
    const unsigned bal = __ballot_sync(0xffffffffu, k);
    if (lane == 0) warp_tot[warp] = __popc(bal);
    __syncthreads();
    int32_t before = 0, total = 0;
#pragma unroll
    for (int w = 0; w < kSelThreads / 32; ++w) {
      before += (w < warp) ? warp_tot[w] : 0;
      total += warp_tot[w];
    }
    const int32_t base = base_s;
    if (k) out[base + before + __popc(bal & ((1u << lane) - 1u))] = static_cast<int32_t>(pos);
    __syncthreads();
    if (threadIdx.x == 0) base_s = base + total;
    __syncthreads();
  }
}

}  // namespace
}  // namespace ssm

extern "C" {

ssm_status ssm_suffix_count(const ssm_suffix_cfg* cfg, int32_t* h_n_local, int32_t* h_n_mid,
                            int32_t* h_n_tail) {
  const ssm_status s = ssm::check_cfg(cfg);
  if (s != SSM_OK) return s;
  int32_t a, b, c;
  ssm::host_counts(*cfg, &a, &b, &c);
  if (h_n_local) *h_n_local = a;
  if (h_n_mid) *h_n_mid = b;
  if (h_n_tail) *h_n_tail = c;
  return SSM_OK;
}

ssm_status ssm_select_suffix_batch(const ssm_suffix_cfg* h_cfgs, int32_t n, int32_t* positions,
                                   int64_t capacity, int64_t* h_offsets, ssm_stream_t stream) {
  if (n < 0 || (n > 0 && !h_cfgs) || capacity < 0) return SSM_ERR_INVALID_ARG;
  std::vector<int64_t> off(static_cast<size_t>(n) + 1, 0);
  for (int32_t i = 0; i < n; ++i) {
    const ssm_status s = ssm::check_cfg(&h_cfgs[i]);
    if (s != SSM_OK) return s;
    int32_t a, b, c;
    ssm::host_counts(h_cfgs[i], &a, &b, &c);
    off[i + 1] = off[i] + a + b + c;
  }
  if (h_offsets)
    for (int32_t i = 0; i <= n; ++i) h_offsets[i] = off[i];
  if (off[n] > capacity) return SSM_ERR_CAPACITY;
  if (off[n] > 0 && !positions) return SSM_ERR_INVALID_ARG;
  for (int32_t first = 0; first < n; first += ssm::kSelMaxPerLaunch) {
    const int32_t cnt = std::min(ssm::kSelMaxPerLaunch, n - first);
    ssm::SelectBatch sb{};
    for (int32_t i = 0; i < cnt; ++i) {
      sb.cfg[i] = h_cfgs[first + i];
      sb.offset[i] = off[first + i];
    }
    ssm::launch_k(ssm::select_kernel, dim3(cnt), dim3(ssm::kSelThreads), 0, reinterpret_cast<cudaStream_t>(stream),
             sb, positions);
    const ssm_status ls = ssm::launch_status();
    if (ls != SSM_OK) return ls;
  }
  return SSM_OK;
}

ssm_status ssm_select_suffix(const ssm_suffix_cfg* cfg, int32_t* positions, int32_t capacity,
                             int32_t* h_count, ssm_stream_t stream) {
  const ssm_status s = ssm::check_cfg(cfg);
  if (s != SSM_OK) return s;
  int32_t a, b, c;
  ssm::host_counts(*cfg, &a, &b, &c);
  if (h_count) *h_count = a + b + c;
  if (capacity < a + b + c) return SSM_ERR_CAPACITY;
  int64_t off[2];
  return ssm_select_suffix_batch(cfg, 1, positions, capacity, off, stream);
}

}  // extern "C"
