// topk.cuh -- pieces of the suffix top-k pass (topk.cu: the k most probable tokens
// of a row and their full-vocabulary probabilities, Sec. 3.2 "Soft Suffix Embedding
// Mixing"): per-thread decreasing candidate lists, the warp merge of those lists,
// the CTA-wide k-th largest of the threads' maxima, and the (max, sum) merge.
#pragma once

#include <cstdint>

#include "sm100_ptx.cuh"

namespace ssm {
namespace topk {

constexpr int kTopMax = 8;                 // list length kept (k <= 8)
constexpr int kTopThreads = 256;
constexpr int kTopStageBytes = 16384;      // one chunk: 64 bytes per thread
constexpr int kTopStages = 2;
constexpr int kTopVecPerThread = kTopStageBytes / 16 / kTopThreads;  // 4
constexpr float kLog2eT = 1.4426950408889634f;
constexpr int64_t kTopMaxSmem = 200 * 1024;   // dynamic shared memory cap: bf16 rows up to 2,744,320 entries, fp32 684,032

__device__ __forceinline__ float ex2t(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

// (a, ia) ranks before (b, ib): larger value, or equal value and lower id.
__device__ __forceinline__ bool better(float a, int ia, float b, int ib) { return a > b || (a == b && ia < ib); }

// Inserts (x, ix) into a decreasing list if it ranks before the last entry.
__device__ __forceinline__ void list_insert(float (&v)[kTopMax], int (&id)[kTopMax], float x, int ix) {
#pragma unroll
  for (int j = kTopMax - 1; j > 0; --j) {
    const bool above = better(x, ix, v[j - 1], id[j - 1]);
    const bool here = better(x, ix, v[j], id[j]);
    const float nv = above ? v[j - 1] : (here ? x : v[j]);
    const int ni = above ? id[j - 1] : (here ? ix : id[j]);
    v[j] = nv;
    id[j] = ni;
  }
  if (better(x, ix, v[0], id[0])) {
    v[0] = x;
    id[0] = ix;
  }
}

// Each warp's k best (value, id) among its lanes' decreasing lists of L entries
// (k rounds of warp argmax over the heads; the winning lane pops its head),
// written to wv / wi [warp][kTopMax].  The caller synchronises before reading.
template <int L>
__device__ __forceinline__ void warp_topk(const float (&lv)[L], const int (&li)[L], int k, float* wv, int* wi) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  float cv[L];
  int ci[L];
#pragma unroll
  for (int j = 0; j < L; ++j) {
    cv[j] = lv[j];
    ci[j] = li[j];
  }
  for (int r = 0; r < k; ++r) {
    float bv = cv[0];
    int bi = ci[0], bl = lane;
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) {
      const float ov = __shfl_xor_sync(0xffffffffu, bv, d);
      const int oi = __shfl_xor_sync(0xffffffffu, bi, d);
      const int ol = __shfl_xor_sync(0xffffffffu, bl, d);
      if (better(ov, oi, bv, bi) || (ov == bv && oi == bi && ol < bl)) {
        bv = ov;
        bi = oi;
        bl = ol;
      }
    }
    if (lane == 0) {
      wv[warp * kTopMax + r] = bv;
      wi[warp * kTopMax + r] = bi;
    }
    if (lane == bl) {
#pragma unroll
      for (int j = 0; j + 1 < L; ++j) {
        cv[j] = cv[j + 1];
        ci[j] = ci[j + 1];
      }
      cv[L - 1] = -INFINITY;
      ci[L - 1] = INT_MAX;
    }
  }
}

__device__ __forceinline__ void ms_merge(float& m, float& s, float m2, float s2) {
  const float mm = fmaxf(m, m2);
  const float a = (s > 0.f) ? s * ex2t((m - mm) * kLog2eT) : 0.f;
  const float b = (s2 > 0.f) ? s2 * ex2t((m2 - mm) * kLog2eT) : 0.f;
  m = mm;
  s = a + b;
}

// Order-preserving map of a float to an unsigned key (larger float, larger key).
__device__ __forceinline__ uint32_t float_key(float x) {
  const uint32_t b = __float_as_uint(x);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}
__device__ __forceinline__ float key_float(uint32_t key) {
  return __uint_as_float((key & 0x80000000u) ? (key & 0x7FFFFFFFu) : ~key);
}

// The k-th largest (with multiplicity) and the largest of the CTA's 256 values
// x, for every thread (one barrier; red holds 8 x kTopMax keys and must not be
// rewritten before the CTA's next barrier).  Each warp writes its k largest
// keys by rounds of warp max, each round taking the lanes that hold the
// maximum; then every warp takes the k-th largest of the written keys the same way.
__device__ __forceinline__ float block_kth(float x, int k, float& top, uint32_t* red) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint32_t key = float_key(x);
  for (int above = 0; above < k;) {
    const uint32_t mx = __reduce_max_sync(0xffffffffu, key);
    const uint32_t ball = __ballot_sync(0xffffffffu, key == mx);
    if (key == mx) {
      const int slot = above + __popc(ball & ((1u << lane) - 1u));
      if (slot < k) red[warp * kTopMax + slot] = mx;
      key = 0u;
    }
    above += __popc(ball);
  }
  __syncthreads();
  // lane l holds slots 2l and 2l + 1 of the 8 x kTopMax table (slots >= k unused: key 0)
  uint32_t a = ((2 * lane) % kTopMax < k) ? red[2 * lane] : 0u;
  uint32_t b = ((2 * lane + 1) % kTopMax < k) ? red[2 * lane + 1] : 0u;
  uint32_t res = 0u;
  for (int above = 0, r = 0; above < k; ++r) {
    const uint32_t mx = __reduce_max_sync(0xffffffffu, max(a, b));
    if (r == 0) top = key_float(mx);
    above += __popc(__ballot_sync(0xffffffffu, a == mx)) + __popc(__ballot_sync(0xffffffffu, b == mx));
    res = mx;
    if (a == mx) a = 0u;
    if (b == mx) b = 0u;
  }
  return key_float(res);
}

}  // namespace topk
}  // namespace ssm
