// topk.cu -- the next step's soft-embedding candidates of the retained suffix
// positions (Sec. 3.2 "Soft Suffix Embedding Mixing": the set T^i_{t+1} of the
// k most probable tokens and their probabilities p^i_{t+1}(v), which Eq. 6
// renormalizes at the next step).  Each row of logits gives its k best token
// ids (ties: lower id first) and their full-vocabulary softmax probabilities.
//
// topk_row_kernel: the unmasking pass's streaming scheme (stream.cuh), one
// row per CTA at a time, read once; the few slices that can hold a candidate
// are re-read at the row's end (see the kernel).
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <type_traits>

#include "common.cuh"
#include "sm100_ptx.cuh"
#include "stream.cuh"
#include "topk.cuh"

namespace ssm {
namespace {

using namespace topk;

__device__ __forceinline__ uint32_t bmax2(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

// A thread's 64 bytes of one chunk are 16 words w[4u + q] (its vector u, word q);
// entry h of word (u, q) is  chunk_start + (u * threads + thread) * epv + q * (epv / 4) + h.
template <typename T>
__device__ __forceinline__ float words_max(const uint32_t (&w)[16]) {
  if constexpr (sizeof(T) == 2) {
    uint32_t x[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) x[c] = bmax2(bmax2(w[c], w[4 + c]), bmax2(w[8 + c], w[12 + c]));
    const uint32_t y = bmax2(bmax2(x[0], x[1]), bmax2(x[2], x[3]));
    return fmaxf(lo_bf16(y), hi_bf16(y));
  } else {
    float a = fmax3(__uint_as_float(w[0]), __uint_as_float(w[1]), __uint_as_float(w[2]));
    float b = fmax3(__uint_as_float(w[3]), __uint_as_float(w[4]), __uint_as_float(w[5]));
    a = fmax3(a, __uint_as_float(w[6]), __uint_as_float(w[7]));
    b = fmax3(b, __uint_as_float(w[8]), __uint_as_float(w[9]));
    a = fmax3(a, __uint_as_float(w[10]), __uint_as_float(w[11]));
    b = fmax3(b, __uint_as_float(w[12]), __uint_as_float(w[13]));
    return fmax3(a, b, fmaxf(__uint_as_float(w[14]), __uint_as_float(w[15])));
  }
}

// One CTA per row at a time (rows dealt round-robin to persistent CTAs), the row
// streamed once through the unmasking pass's cp.async ring (stream.cuh).  Each
// thread folds its 64 bytes of a chunk into a running (max m, sum of exp(x - m))
// and records the slice's maximum in shared memory.  At the row's end the CTA
// fixes T = the k-th largest of the threads' maxima: k distinct entries reach T,
// so the row's k-th best value is >= T and only slices whose maximum reaches T
// can hold a candidate (on random logits about k of the row's 4096 slices).  Each
// thread re-reads those of its slices from global memory and keeps a decreasing
// list of its 8 best (value, id) among their entries >= T; each warp then takes
// its k best by k rounds of warp argmax and one thread merges the eight lists.
template <typename T>
__global__ void __launch_bounds__(kTopThreads, 5) topk_row_kernel(const T* __restrict__ logits, int64_t vocab,
                                                              int64_t n_rows, int k, int32_t* __restrict__ ids,
                                                              float* __restrict__ probs) {
  pdl_enter();
  constexpr int ESZ = sizeof(T);
  constexpr int EPV = 16 / ESZ;          // entries per 16-byte vector
  constexpr int EPW = EPV / 4;           // entries per word
  constexpr int EPC = kTopStageBytes / ESZ;   // entries per chunk
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  // [chunk][thread] slice maxima, stored in the logits' own type (exact)
  using Slice = typename std::conditional<ESZ == 2, uint16_t, uint32_t>::type;
  Slice* slice_max = reinterpret_cast<Slice*>(ring + kTopStages * kTopStageBytes);
  // the warps' row states and k-best lists, double-buffered by row parity: warp 0 reads one row's
  // after the CTA barrier while the other warps go on to the next row, which writes the other set
  __shared__ float red_m[2][kTopThreads / 32], red_s[2][kTopThreads / 32];
  __shared__ float red_kv[2][(kTopThreads / 32) * kTopMax];
  __shared__ int red_ki[2][(kTopThreads / 32) * kTopMax];
  __shared__ uint32_t red_key[(kTopThreads / 32) * kTopMax];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t row_bytes = vocab * ESZ;
  const int nchunk = static_cast<int>((row_bytes + kTopStageBytes - 1) / kTopStageBytes);
  const uint32_t ninf = (ESZ == 2) ? 0xFF80FF80u : 0xFF800000u;
  int64_t irow = blockIdx.x;
  int ichunk = 0;
  auto issue = [&](int slot) {
    if (irow < n_rows) {
      const int64_t off = static_cast<int64_t>(ichunk) * kTopStageBytes;
      const uint8_t* src = reinterpret_cast<const uint8_t*>(logits + irow * vocab) + off;
      uint8_t* dst = ring + slot * kTopStageBytes;
#pragma unroll
      for (int u = 0; u < kTopVecPerThread; ++u) {
        const int vi = u * kTopThreads + threadIdx.x;
        if (vi * 16 < row_bytes - off) cp_async16(dst + vi * 16, src + vi * 16);
      }
      if (++ichunk == nchunk) {
        ichunk = 0;
        irow += gridDim.x;
      }
    }
    cp_async_commit();
  };
#pragma unroll
  for (int q = 0; q < kTopStages; ++q) issue(q);

  int slot = 0;
  int par = 0;  // the row's buffer set
  for (int64_t row = blockIdx.x; row < n_rows; row += gridDim.x, par ^= 1) {
    float m = -INFINITY, s = 0.f;
    for (int c = 0; c < nchunk; ++c) {
      cp_async_wait<kTopStages - 1>();
      const int64_t off = static_cast<int64_t>(c) * kTopStageBytes;
      const int chunk_bytes = static_cast<int>(min(static_cast<int64_t>(kTopStageBytes), row_bytes - off));
      const uint4* sv = reinterpret_cast<const uint4*>(ring + slot * kTopStageBytes);
      uint32_t w[16];
#pragma unroll
      for (int u = 0; u < kTopVecPerThread; ++u) {
        const int vi = u * kTopThreads + threadIdx.x;
        const uint4 v = vi * 16 < chunk_bytes ? sv[vi] : make_uint4(ninf, ninf, ninf, ninf);
        w[4 * u] = v.x;
        w[4 * u + 1] = v.y;
        w[4 * u + 2] = v.z;
        w[4 * u + 3] = v.w;
      }
      issue(slot);
      slot = (slot + 1) % kTopStages;
      const float cm = words_max<T>(w);
      slice_max[c * kTopThreads + threadIdx.x] = static_cast<Slice>(__float_as_uint(cm) >> (32 - 8 * ESZ));
      if (cm > m) {
        if (m > -INFINITY) s *= ex2t((m - cm) * kLog2eT);
        m = cm;
      }
      if (m > -INFINITY) {
        const float mb = m * kLog2eT;
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int e = 0; e < 16; e += (ESZ == 2 ? 1 : 2)) {
          float x0, x1;
          if constexpr (ESZ == 2) {
            x0 = lo_bf16(w[e]);
            x1 = hi_bf16(w[e]);
          } else {
            x0 = __uint_as_float(w[e]);
            x1 = __uint_as_float(w[e + 1]);
          }
          float t0, t1;
          ffma2(t0, t1, x0, x1, kLog2eT, kLog2eT, -mb, -mb);
          const int a = (ESZ == 2 ? e : e >> 1) & 3;
          fadd2_acc(sa[a], sb[a], ex2t(t0), ex2t(t1));
        }
        s += ((sa[0] + sb[0]) + (sa[1] + sb[1])) + ((sa[2] + sb[2]) + (sa[3] + sb[3]));
      }
    }
    // T, then the candidates of the slices whose maximum reaches it
    float top;
    const float thr = block_kth(m, k, top, red_key);
    float tv[kTopMax];
    int ti[kTopMax];
#pragma unroll
    for (int j = 0; j < kTopMax; ++j) {
      tv[j] = -INFINITY;
      ti[j] = INT_MAX;
    }
    for (int c = 0; c < nchunk; ++c) {
      if (__uint_as_float(static_cast<uint32_t>(slice_max[c * kTopThreads + threadIdx.x]) << (32 - 8 * ESZ)) < thr)
        continue;
      const int64_t off = static_cast<int64_t>(c) * kTopStageBytes;
      const int chunk_bytes = static_cast<int>(min(static_cast<int64_t>(kTopStageBytes), row_bytes - off));
      const uint4* gv = reinterpret_cast<const uint4*>(reinterpret_cast<const uint8_t*>(logits + row * vocab) + off);
#pragma unroll
      for (int u = 0; u < kTopVecPerThread; ++u) {
        const int vi = u * kTopThreads + threadIdx.x;
        const uint4 v = vi * 16 < chunk_bytes ? __ldg(gv + vi) : make_uint4(ninf, ninf, ninf, ninf);
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
#pragma unroll
          for (int h = 0; h < EPW; ++h) {
            const float f = (ESZ == 2) ? (h ? hi_bf16(w4[q]) : lo_bf16(w4[q])) : __uint_as_float(w4[q]);
            const int id = c * EPC + vi * EPV + q * EPW + h;
            if (f >= thr && better(f, id, tv[kTopMax - 1], ti[kTopMax - 1])) list_insert(tv, ti, f, id);
          }
        }
      }
    }
    // the row's (max, sum) and its k best
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) ms_merge(m, s, __shfl_xor_sync(0xffffffffu, m, d), __shfl_xor_sync(0xffffffffu, s, d));
    if (lane == 0) {
      red_m[par][warp] = m;
      red_s[par][warp] = s;
    }
    warp_topk<kTopMax>(tv, ti, k, red_kv[par], red_ki[par]);
    __syncthreads();
    if (warp == 0) {
      // lanes 0..7 merge the eight warps' (max, sum); every lane then holds the row's
      float rm = lane < kTopThreads / 32 ? red_m[par][lane] : -INFINITY;
      float rs = lane < kTopThreads / 32 ? red_s[par][lane] : 0.f;
#pragma unroll
      for (int d = (kTopThreads / 32) / 2; d >= 1; d >>= 1)
        ms_merge(rm, rs, __shfl_xor_sync(0xffffffffu, rm, d), __shfl_xor_sync(0xffffffffu, rs, d));
      rm = __shfl_sync(0xffffffffu, rm, 0);
      rs = __shfl_sync(0xffffffffu, rs, 0);
      const float inv = 1.f / rs;
      // the k best of the eight lists: lane l holds entries l and l + 32 of the [warp][kTopMax]
      // table (entries past a list's k are unused), then k rounds of warp argmax, the winning
      // entry cleared each round
      constexpr int NE = (kTopThreads / 32) * kTopMax;
      static_assert(NE <= 64, "two list entries per lane");
      const bool u0 = lane % kTopMax < k, u1 = (lane + 32) < NE && (lane + 32) % kTopMax < k;
      float v0 = u0 ? red_kv[par][lane] : -INFINITY, v1 = u1 ? red_kv[par][lane + 32] : -INFINITY;
      int i0 = u0 ? red_ki[par][lane] : INT_MAX, i1 = u1 ? red_ki[par][lane + 32] : INT_MAX;
      for (int r = 0; r < k; ++r) {
        const bool first = better(v0, i0, v1, i1) || !(better(v1, i1, v0, i0));
        float bv = first ? v0 : v1;
        int bi = first ? i0 : i1;
#pragma unroll
        for (int d = 16; d >= 1; d >>= 1) {
          const float ov = __shfl_xor_sync(0xffffffffu, bv, d);
          const int oi = __shfl_xor_sync(0xffffffffu, bi, d);
          if (better(ov, oi, bv, bi)) {
            bv = ov;
            bi = oi;
          }
        }
        // ids are distinct within a row, so exactly one entry holds the winner
        if (i0 == bi) {
          v0 = -INFINITY;
          i0 = INT_MAX;
        } else if (i1 == bi) {
          v1 = -INFINITY;
          i1 = INT_MAX;
        }
        if (lane == 0) {
          ids[row * k + r] = bi;
          probs[row * k + r] = ex2t((bv - rm) * kLog2eT) * inv;
        }
      }
    }
  }
  cp_async_wait<0>();
}

// Opts the kernel into the largest dynamic shared memory any call may ask for, once per device
// (a ceiling: a call's own size decides its occupancy; setting the first call's size would
// make a later call with a longer vocabulary fail to launch).
template <auto kernel>
bool topk_attr_set() {
  constexpr size_t bytes = kTopMaxSmem;
  static std::atomic<uint64_t> done{0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return false;
  const uint64_t bit = 1ull << (dev & 63);
  if (done.load() & bit) return true;
  if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(bytes)) !=
      cudaSuccess)
    return false;
  done.fetch_or(bit);
  return true;
}

}  // namespace
}  // namespace ssm

extern "C" {

ssm_status ssm_suffix_topk(const void* logits, ssm_dtype dtype, int64_t n_rows, int64_t vocab, int32_t k,
                           int32_t* ids, float* probs, ssm_stream_t stream) {
  if (dtype != SSM_DTYPE_BF16 && dtype != SSM_DTYPE_F32) return SSM_ERR_UNSUPPORTED;
  if (n_rows < 0 || vocab <= 0) return SSM_ERR_INVALID_ARG;
  if (k < 1 || k > ssm::kTopMax) return SSM_ERR_UNSUPPORTED;
  if (k > vocab) return SSM_ERR_INVALID_ARG;
  if (vocab > INT32_MAX) return SSM_ERR_UNSUPPORTED;
  if (n_rows == 0) return SSM_OK;
  if (!logits || !ids || !probs) return SSM_ERR_INVALID_ARG;
  const int esz = dtype == SSM_DTYPE_BF16 ? 2 : 4;
  // 16-byte copies need 16-byte aligned rows
  if (!ssm::aligned16(logits) || (vocab * esz) % 16 != 0) return SSM_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  // the ring plus one logit per (chunk, thread): the row's slice maxima
  const int64_t nchunk = (vocab * esz + ssm::kTopStageBytes - 1) / ssm::kTopStageBytes;
  const int64_t smem64 = ssm::kTopStages * ssm::kTopStageBytes + nchunk * ssm::kTopThreads * esz + 128;
  if (smem64 > ssm::kTopMaxSmem) return SSM_ERR_UNSUPPORTED;
  const size_t smem = static_cast<size_t>(smem64);
  const int grid = static_cast<int>(std::min<int64_t>(n_rows, 5ll * ssm::num_sms()));
  if (dtype == SSM_DTYPE_BF16) {
    if (!ssm::topk_attr_set<ssm::topk_row_kernel<__nv_bfloat16>>()) return SSM_ERR_CUDA;
    ssm::launch_k(ssm::topk_row_kernel<__nv_bfloat16>, dim3(grid), dim3(ssm::kTopThreads), smem, st,
             static_cast<const __nv_bfloat16*>(logits), vocab, n_rows, k, ids, probs);
  } else {
    if (!ssm::topk_attr_set<ssm::topk_row_kernel<float>>()) return SSM_ERR_CUDA;
    ssm::launch_k(ssm::topk_row_kernel<float>, dim3(grid), dim3(ssm::kTopThreads), smem, st,
             static_cast<const float*>(logits), vocab,
                                                                     n_rows, k, ids, probs);
  }
  return ssm::launch_status();
}

}  // extern "C"
