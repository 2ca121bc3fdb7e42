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

namespace ssm {
namespace {

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

// The k best of the eight warps' lists in wv / wi (k rounds over their heads);
// returns the k-th value, sets top to the best one and, if out_v is given,
// writes the k (value, id).
__device__ __forceinline__ float merge_warp_lists(const float* wv, const int* wi, int k, float& top, float* out_v,
                                                  int* out_i) {
  int head[kTopThreads / 32];
#pragma unroll
  for (int w = 0; w < kTopThreads / 32; ++w) head[w] = 0;
  float t = -INFINITY;
  for (int r = 0; r < k; ++r) {
    int bw = 0;
    float bv = -INFINITY;
    int bi = INT_MAX;
#pragma unroll
    for (int w = 0; w < kTopThreads / 32; ++w) {
      if (head[w] < k) {
        const float v = wv[w * kTopMax + head[w]];
        const int i = wi[w * kTopMax + head[w]];
        if (better(v, i, bv, bi)) {
          bv = v;
          bi = i;
          bw = w;
        }
      }
    }
#pragma unroll
    for (int w = 0; w < kTopThreads / 32; ++w) head[w] += (w == bw) ? 1 : 0;
    if (out_v) {
      out_v[r] = bv;
      out_i[r] = bi;
    }
    if (r == 0) top = bv;
    t = bv;
  }
  return t;
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
__global__ void __launch_bounds__(kTopThreads) topk_row_kernel(const T* __restrict__ logits, int64_t vocab,
                                                              int64_t n_rows, int k, int32_t* __restrict__ ids,
                                                              float* __restrict__ probs) {
  constexpr int ESZ = sizeof(T);
  constexpr int EPV = 16 / ESZ;          // entries per 16-byte vector
  constexpr int EPW = EPV / 4;           // entries per word
  constexpr int EPC = kTopStageBytes / ESZ;   // entries per chunk
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  // [chunk][thread] slice maxima, stored in the logits' own type (exact)
  using Slice = typename std::conditional<ESZ == 2, uint16_t, uint32_t>::type;
  Slice* slice_max = reinterpret_cast<Slice*>(ring + kTopStages * kTopStageBytes);
  __shared__ float red_m[kTopThreads / 32], red_s[kTopThreads / 32];
  __shared__ float red_kv[(kTopThreads / 32) * kTopMax];
  __shared__ int red_ki[(kTopThreads / 32) * kTopMax];
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
  for (int64_t row = blockIdx.x; row < n_rows; row += gridDim.x) {
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
      red_m[warp] = m;
      red_s[warp] = s;
    }
    warp_topk<kTopMax>(tv, ti, k, red_kv, red_ki);
    __syncthreads();
    if (threadIdx.x == 0) {
      float rm = red_m[0], rs = red_s[0];
      for (int q = 1; q < kTopThreads / 32; ++q) ms_merge(rm, rs, red_m[q], red_s[q]);
      const float inv = 1.f / rs;
      float bv[kTopMax], best;
      int bi[kTopMax];
      merge_warp_lists(red_kv, red_ki, k, best, bv, bi);
      for (int r = 0; r < k; ++r) {
        ids[row * k + r] = bi[r];
        probs[row * k + r] = ex2t((bv[r] - rm) * kLog2eT) * inv;
      }
    }
    __syncthreads();
  }
  cp_async_wait<0>();
}

template <auto kernel>
bool topk_attr_set(size_t bytes) {
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
    if (!ssm::topk_attr_set<ssm::topk_row_kernel<__nv_bfloat16>>(smem)) return SSM_ERR_CUDA;
    ssm::topk_row_kernel<__nv_bfloat16><<<grid, ssm::kTopThreads, smem, st>>>(
        static_cast<const __nv_bfloat16*>(logits), vocab, n_rows, k, ids, probs);
  } else {
    if (!ssm::topk_attr_set<ssm::topk_row_kernel<float>>(smem)) return SSM_ERR_CUDA;
    ssm::topk_row_kernel<float><<<grid, ssm::kTopThreads, smem, st>>>(static_cast<const float*>(logits), vocab,
                                                                     n_rows, k, ids, probs);
  }
  return ssm::launch_status();
}

}  // extern "C"
