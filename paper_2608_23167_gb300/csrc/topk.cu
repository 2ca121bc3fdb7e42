// topk.cu -- the next step's soft-embedding candidates of the retained suffix
// positions (Sec. 3.2 "Soft Suffix Embedding Mixing": the set T^i_{t+1} of the
// k most probable tokens and their probabilities p^i_{t+1}(v), which Eq. 6
// renormalizes at the next step).  Each row of logits gives its k best token
// ids (ties: lower id first) and their full-vocabulary softmax probabilities.
//
// topk_row_kernel: the unmasking pass's streaming scheme (stream.cuh), one
// row per CTA at a time, with a threshold that keeps the candidate lists idle
// after the row's first chunk (see the kernel).
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>

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

__device__ __forceinline__ void ms_merge(float& m, float& s, float m2, float s2) {
  const float mm = fmaxf(m, m2);
  const float a = (s > 0.f) ? s * ex2t((m - mm) * kLog2eT) : 0.f;
  const float b = (s2 > 0.f) ? s2 * ex2t((m2 - mm) * kLog2eT) : 0.f;
  m = mm;
  s = a + b;
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
// returns the k-th value and, if out_v is given, writes the k (value, id).
__device__ __forceinline__ float merge_warp_lists(const float* wv, const int* wi, int k, float* out_v,
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
    t = bv;
  }
  return t;
}

// The row's k-th best value so far among all lanes' lists, as a lower bound:
// every thread of the CTA gets it (one barrier pair).
template <int L>
__device__ __forceinline__ float block_kth(const float (&lv)[L], const int (&li)[L], int k, float* wv, int* wi) {
  warp_topk<L>(lv, li, k, wv, wi);
  __syncthreads();
  const float t = merge_warp_lists(wv, wi, k, nullptr, nullptr);
  __syncthreads();
  return t;
}

// One CTA per row at a time (rows dealt round-robin to persistent CTAs).  The
// row streams through the cp.async ring; every thread keeps (max, sum of exp)
// and a decreasing list of its 8 best (value, id).  A threshold T bounds the
// row's k-th best value from below: first the k-th largest of the threads'
// maxima of chunk 0, then, after chunks 1 and 3, the k-th best entry of all
// lists (k distinct entries of the row reach it either way).  Nothing below T
// can be a candidate, and a chunk touches a list only for a value >= T that
// ranks before the list's last entry, which soon becomes rare.  At the
// row's end each warp takes its k best by k rounds of warp argmax and one
// thread merges the eight lists.
template <typename T>
__global__ void __launch_bounds__(kTopThreads) topk_row_kernel(const T* __restrict__ logits, int64_t vocab,
                                                              int64_t n_rows, int k, int32_t* __restrict__ ids,
                                                              float* __restrict__ probs) {
  constexpr int ESZ = sizeof(T);
  constexpr int EPV = 16 / ESZ;                       // elements per 16-byte vector
  constexpr int PER = kTopVecPerThread * EPV;         // values per thread and chunk
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  __shared__ float red_m[kTopThreads / 32], red_s[kTopThreads / 32];
  __shared__ float red_kv[(kTopThreads / 32) * kTopMax];
  __shared__ int red_ki[(kTopThreads / 32) * kTopMax];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  ChunkIter is{static_cast<int64_t>(blockIdx.x) - gridDim.x, 0, 0, 0, 0, false};
  chunk_seek<T>(is, vocab, vocab, 1, n_rows, nullptr);
  auto issue = [&](int slot) {
    if (is.valid) {
      const uint8_t* src = reinterpret_cast<const uint8_t*>(logits + is.row * vocab) + is.off;
      uint8_t* dst = ring + slot * kTopStageBytes;
#pragma unroll
      for (int u = 0; u < kTopVecPerThread; ++u) {
        const int vi = u * kTopThreads + threadIdx.x;
        if (vi * 16 < is.bytes - is.off) cp_async16(dst + vi * 16, src + vi * 16);
      }
      is.off += kTopStageBytes;
      chunk_seek<T>(is, vocab, vocab, 1, n_rows, nullptr);
    }
    cp_async_commit();
  };
#pragma unroll
  for (int q = 0; q < kTopStages; ++q) issue(q);

  ChunkIter cs{static_cast<int64_t>(blockIdx.x) - gridDim.x, 0, 0, 0, 0, false};
  chunk_seek<T>(cs, vocab, vocab, 1, n_rows, nullptr);
  int slot = 0;
  while (cs.valid) {
    const int64_t row = cs.item;
    float m = -INFINITY, s = 0.f, thr = -INFINITY;
    float tv[kTopMax];
    int ti[kTopMax];
#pragma unroll
    for (int j = 0; j < kTopMax; ++j) {
      tv[j] = -INFINITY;
      ti[j] = INT_MAX;
    }
    int nchunk = 0;  // chunks of this row done
    while (cs.valid && cs.item == row) {
      cp_async_wait<kTopStages - 1>();
      const int chunk_bytes = static_cast<int>(min(static_cast<int64_t>(kTopStageBytes), cs.bytes - cs.off));
      const uint4* sv = reinterpret_cast<const uint4*>(ring + slot * kTopStageBytes);
      const uint32_t ninf = (ESZ == 2) ? 0xFF80FF80u : 0xFF800000u;
      float f[PER];
#pragma unroll
      for (int u = 0; u < kTopVecPerThread; ++u) {
        const int vi = u * kTopThreads + threadIdx.x;
        const uint4 v = vi * 16 < chunk_bytes ? sv[vi] : make_uint4(ninf, ninf, ninf, ninf);
        const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if constexpr (ESZ == 2) {
            f[u * 8 + 2 * q] = lo_bf16(w4[q]);
            f[u * 8 + 2 * q + 1] = hi_bf16(w4[q]);
          } else {
            f[u * 4 + q] = __uint_as_float(w4[q]);
          }
        }
      }
      float c4[4] = {f[0], f[1], f[2], f[3]};
#pragma unroll
      for (int e = 4; e < PER; e += 8) {
        c4[0] = fmax3(c4[0], f[e], f[e + 1]);
        c4[1] = fmax3(c4[1], f[e + 2], f[e + 3]);
        if (e + 4 < PER) {
          c4[2] = fmax3(c4[2], f[e + 4], f[e + 5]);
          c4[3] = fmax3(c4[3], f[e + 6], f[e + 7]);
        }
      }
      const float cm = fmaxf(fmaxf(c4[0], c4[1]), fmaxf(c4[2], c4[3]));
      if (nchunk == 0) {
        // before any list work: T = the k-th largest of the threads' chunk maxima
        const float one[1] = {cm};
        const int tag[1] = {static_cast<int>(threadIdx.x)};   // distinct per thread: only the value is used
        thr = block_kth<1>(one, tag, k, red_kv, red_ki);
      }
      // a value enters the list only when it reaches the threshold and ranks before the
      // list's last entry
      if (cm >= thr && cm >= tv[kTopMax - 1]) {
        const int tbase = static_cast<int>(cs.off / ESZ) + static_cast<int>(threadIdx.x) * EPV;
        // scan only the max chains whose maximum qualifies (chain q holds e = q and the pairs
        // 4 + 8i + 2q, 5 + 8i + 2q of the reduction above); chains are visited out of id
        // order, so an entry is compared with the list's last one by (value, id)
#pragma unroll
        for (int q = 0; q < 4; ++q) {
          if (c4[q] >= thr && c4[q] >= tv[kTopMax - 1]) {
#pragma unroll
            for (int e = 0; e < PER; ++e) {
              const bool in_chain = (e < 4) ? (e == q) : (((e - 4) % 8) / 2 == q);
              const int id = tbase + (e / EPV) * kTopThreads * EPV + (e % EPV);
              if (in_chain && f[e] >= thr && better(f[e], id, tv[kTopMax - 1], ti[kTopMax - 1]))
                list_insert(tv, ti, f[e], id);
            }
          }
        }
      }
      if (cm > m) {
        if (m > -INFINITY) s *= ex2t((m - cm) * kLog2eT);
        m = cm;
      }
      if (m > -INFINITY) {
        const float mb = m * kLog2eT;
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int e = 0; e < PER; e += 2) {
          float t0, t1;
          ffma2(t0, t1, f[e], f[e + 1], kLog2eT, kLog2eT, -mb, -mb);
          fadd2_acc(sa[(e >> 1) & 3], sb[(e >> 1) & 3], ex2t(t0), ex2t(t1));
        }
        s += ((sa[0] + sb[0]) + (sa[1] + sb[1])) + ((sa[2] + sb[2]) + (sa[3] + sb[3]));
      }
      issue(slot);
      slot = (slot + 1) % kTopStages;
      cs.off += kTopStageBytes;
      if (cs.off >= cs.bytes) chunk_seek<T>(cs, vocab, vocab, 1, n_rows, nullptr);
      if (nchunk == 1 || nchunk == 3) thr = fmaxf(thr, block_kth<kTopMax>(tv, ti, k, red_kv, red_ki));
      ++nchunk;
    }
    // the row's (max, sum)
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) ms_merge(m, s, __shfl_xor_sync(0xffffffffu, m, d), __shfl_xor_sync(0xffffffffu, s, d));
    if (lane == 0) {
      red_m[warp] = m;
      red_s[warp] = s;
    }
    // the row's k best: the warps' k best, then thread 0 merges them
    warp_topk<kTopMax>(tv, ti, k, red_kv, red_ki);
    __syncthreads();
    if (threadIdx.x == 0) {
      float rm = red_m[0], rs = red_s[0];
      for (int w = 1; w < kTopThreads / 32; ++w) ms_merge(rm, rs, red_m[w], red_s[w]);
      const float inv = 1.f / rs;
      float bv[kTopMax];
      int bi[kTopMax];
      merge_warp_lists(red_kv, red_ki, k, bv, bi);
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
  const size_t smem = ssm::kTopStages * ssm::kTopStageBytes + 128;
  const int grid = static_cast<int>(std::min<int64_t>(n_rows, 6ll * ssm::num_sms()));
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
