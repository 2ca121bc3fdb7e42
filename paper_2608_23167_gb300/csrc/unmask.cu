// unmask.cu -- confidence-based unmasking (Sec. 4.1 "Baselines": Vanilla top-1
// and parallel threshold decoding; Sec. 4.5: margin decoding).
//
// Pass 1 (unmask_partial_kernel): every masked row of logits is cut into
// chunks; one CTA reads one chunk once with 16-byte loads and reduces it to
// (max, sum of exp(x - max), first argmax, second-largest logit).  The grid is
// chunks x rows, so a 126464-entry bf16 row spreads over 16 CTAs and the whole
// read is spread evenly over the SMs.  Pass 2 (unmask_commit_kernel): one CTA
// per batch row merges the chunk partials of its positions, writes conf /
// argmax / p2 and applies the commit rule.  Logits of unmasked rows are never
// read.
#include <cuda_bf16.h>

#include <mutex>

#include "common.cuh"

namespace ssm {
namespace {

constexpr int kUnmaskThreads = 256;
constexpr int kUnroll = 16;                        // 16-byte vectors per thread per chunk
constexpr float kLog2e = 1.4426950408889634f;

struct Partial {
  float m;    // max logit
  float s;    // sum of exp(x - m)
  int idx;    // lowest index holding m
  float m2;   // second-largest logit (a tied max counts twice)
};

__device__ __forceinline__ float ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ void observe(float x, int i, float& m, int& idx, float& m2) {
  if (x > m) {
    m2 = m;
    m = x;
    idx = i;
  } else if (x > m2) {
    m2 = x;
  }
}

__device__ __forceinline__ Partial merge(const Partial& a, const Partial& b) {
  Partial r;
  if (a.m > b.m) {
    r.m = a.m;
    r.idx = a.idx;
    r.m2 = fmaxf(a.m2, b.m);
  } else if (b.m > a.m) {
    r.m = b.m;
    r.idx = b.idx;
    r.m2 = fmaxf(b.m2, a.m);
  } else {
    r.m = a.m;
    r.idx = min(a.idx, b.idx);
    r.m2 = a.m;
  }
  const float sa = (a.s > 0.f) ? a.s * ex2((a.m - r.m) * kLog2e) : 0.f;
  const float sb = (b.s > 0.f) ? b.s * ex2((b.m - r.m) * kLog2e) : 0.f;
  r.s = sa + sb;
  return r;
}

__device__ __forceinline__ Partial shfl_partial(const Partial& p, int delta) {
  Partial q;
  q.m = __shfl_xor_sync(0xffffffffu, p.m, delta);
  q.s = __shfl_xor_sync(0xffffffffu, p.s, delta);
  q.idx = __shfl_xor_sync(0xffffffffu, p.idx, delta);
  q.m2 = __shfl_xor_sync(0xffffffffu, p.m2, delta);
  return q;
}

template <typename T>
struct Vec;
template <>
struct Vec<__nv_bfloat16> {
  static constexpr int N = 8;
  __device__ static void unpack(const uint4& v, float (&f)[8]) {
    const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      f[2 * i] = __uint_as_float(w[i] << 16);
      f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
    }
  }
  __device__ static float scalar(const __nv_bfloat16* p, int64_t i) { return __bfloat162float(p[i]); }
};
template <>
struct Vec<float> {
  static constexpr int N = 4;
  __device__ static void unpack(const uint4& v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
  }
  __device__ static float scalar(const float* p, int64_t i) { return p[i]; }
};

// Block-wide reductions over the 256 threads of a CTA (result in every thread).
__device__ __forceinline__ float block_max(float v, float* red) {
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, d));
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = v;
  __syncthreads();
  v = red[lane & (kUnmaskThreads / 32 - 1)];
#pragma unroll
  for (int d = kUnmaskThreads / 64; d >= 1; d >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, d));
  return v;
}

// Chunk of one row: thread t holds vectors t, t + 256, ..., t + 256 (U - 1) of
// the chunk (16 bytes each, so a warp reads 512 contiguous bytes per vector).
// Pass 1 keeps the two largest values per thread; after the block maximum M is
// known, pass 2 sums exp(x - M) and the holder(s) of M report its first index.
template <typename T, int U>
__global__ void __launch_bounds__(kUnmaskThreads) unmask_partial_vec_kernel(
    const T* __restrict__ logits, int64_t vocab, int64_t chunk, int n_chunks,
    const uint8_t* __restrict__ masked, Partial* __restrict__ part) {
  constexpr int N = Vec<T>::N;
  __shared__ float red_f[kUnmaskThreads / 32];
  __shared__ Partial red_p[kUnmaskThreads / 32];
  const int64_t row = blockIdx.y;
  if (!masked[row]) return;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * chunk;
  const int64_t c1 = min(vocab, c0 + chunk);
  const uint4* xv = reinterpret_cast<const uint4*>(logits + row * vocab);
  uint4 v[U];
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int64_t e = c0 + (static_cast<int64_t>(u) * kUnmaskThreads + threadIdx.x) * N;
    v[u] = (e < c1) ? __ldcs(xv + e / N) : make_uint4(0, 0, 0, 0);
  }
  float m1 = -INFINITY, m2 = -INFINITY;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int64_t e = c0 + (static_cast<int64_t>(u) * kUnmaskThreads + threadIdx.x) * N;
    if (e < c1) {
      float f[N];
      Vec<T>::unpack(v[u], f);
#pragma unroll
      for (int c = 0; c < N; ++c) {
        m2 = fmaxf(m2, fminf(m1, f[c]));
        m1 = fmaxf(m1, f[c]);
      }
    }
  }
  const float M = block_max(m1, red_f);
  const float mb = (M == -INFINITY) ? 0.f : M * kLog2e;  // a chunk of -inf logits sums to 0
  float s = 0.f;
  int idx = INT_MAX;
#pragma unroll
  for (int u = 0; u < U; ++u) {
    const int64_t e = c0 + (static_cast<int64_t>(u) * kUnmaskThreads + threadIdx.x) * N;
    if (e < c1) {
      float f[N];
      Vec<T>::unpack(v[u], f);
#pragma unroll
      for (int c = 0; c < N; ++c) s += ex2(fmaf(f[c], kLog2e, -mb));
      if (m1 == M && idx == INT_MAX) {
#pragma unroll
        for (int c = 0; c < N; ++c)
          if (f[c] == M && idx == INT_MAX) idx = static_cast<int>(e + c);
      }
    }
  }
  // (m, s, idx, second): a thread whose maximum is below M offers it as a second
  // candidate; two threads holding M make M itself the second-largest value.
  Partial p{M, s, idx, (m1 == M) ? m2 : m1};
  int holders = (m1 == M) ? 1 : 0;
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) {
    p.s += __shfl_xor_sync(0xffffffffu, p.s, d);
    p.idx = min(p.idx, __shfl_xor_sync(0xffffffffu, p.idx, d));
    p.m2 = fmaxf(p.m2, __shfl_xor_sync(0xffffffffu, p.m2, d));
    holders += __shfl_xor_sync(0xffffffffu, holders, d);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) {
    p.m = __int_as_float(holders);  // the warp's holder count rides in the unused m field
    red_p[warp] = p;
  }
  __syncthreads();
  if (warp == 0) {
    Partial q = red_p[lane & (kUnmaskThreads / 32 - 1)];
    int h = (lane < kUnmaskThreads / 32) ? __float_as_int(q.m) : 0;
    if (lane >= kUnmaskThreads / 32) q = Partial{0.f, 0.f, INT_MAX, -INFINITY};
#pragma unroll
    for (int d = kUnmaskThreads / 64; d >= 1; d >>= 1) {
      q.s += __shfl_xor_sync(0xffffffffu, q.s, d);
      q.idx = min(q.idx, __shfl_xor_sync(0xffffffffu, q.idx, d));
      q.m2 = fmaxf(q.m2, __shfl_xor_sync(0xffffffffu, q.m2, d));
      h += __shfl_xor_sync(0xffffffffu, h, d);
    }
    if (lane == 0) part[row * n_chunks + blockIdx.x] = Partial{M, q.s, q.idx, (h >= 2) ? M : q.m2};
  }
}

// Rows whose length or alignment rules out 16-byte vectors: one element per
// thread per step, online (max, second, first index) then the exp sum.
template <typename T>
__global__ void __launch_bounds__(kUnmaskThreads) unmask_partial_scalar_kernel(
    const T* __restrict__ logits, int64_t vocab, int64_t chunk, int n_chunks,
    const uint8_t* __restrict__ masked, Partial* __restrict__ part) {
  const int64_t row = blockIdx.y;
  if (!masked[row]) return;
  const int64_t c0 = static_cast<int64_t>(blockIdx.x) * chunk;
  const int64_t c1 = min(vocab, c0 + chunk);
  const T* x = logits + row * vocab;
  float m = -INFINITY, m2 = -INFINITY;
  int idx = INT_MAX;
  float s = 0.f;
  for (int64_t e = c0 + threadIdx.x; e < c1; e += kUnmaskThreads)
    observe(Vec<T>::scalar(x, e), static_cast<int>(e), m, idx, m2);
  if (m > -INFINITY) {
    const float mb = m * kLog2e;
    for (int64_t e = c0 + threadIdx.x; e < c1; e += kUnmaskThreads)
      s += ex2(fmaf(Vec<T>::scalar(x, e), kLog2e, -mb));
  }
  Partial p{m, s, idx, m2};
#pragma unroll
  for (int d = 16; d >= 1; d >>= 1) p = merge(p, shfl_partial(p, d));
  __shared__ Partial sp[kUnmaskThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) sp[warp] = p;
  __syncthreads();
  if (warp == 0) {
    p = (lane < kUnmaskThreads / 32) ? sp[lane] : Partial{-INFINITY, 0.f, INT_MAX, -INFINITY};
#pragma unroll
    for (int d = 4; d >= 1; d >>= 1) p = merge(p, shfl_partial(p, d));
    if (lane == 0) part[row * n_chunks + blockIdx.x] = p;
  }
}

// One CTA per batch row; thread j owns block position j.
__global__ void __launch_bounds__(1024) unmask_commit_kernel(
    int block_len, int n_chunks, const uint8_t* __restrict__ masked, const Partial* __restrict__ part,
    int mode, float threshold, int topk, int min_commit, float* __restrict__ conf,
    int32_t* __restrict__ argmax, float* __restrict__ p2_out, uint8_t* __restrict__ commit) {
  extern __shared__ float smem[];
  float* s_conf = smem;                                               // [block_len]
  float* s_score = smem + block_len;                                  // [block_len]
  uint8_t* s_masked = reinterpret_cast<uint8_t*>(smem + 2 * block_len);  // [block_len]
  uint8_t* s_pass = s_masked + block_len;                             // [block_len]
  __shared__ int s_npass;
  const int64_t b = blockIdx.x;
  const int j = threadIdx.x;
  if (j == 0) s_npass = 0;
  float cj = 0.f, p2 = 0.f;
  int aj = -1;
  bool mj = false;
  if (j < block_len) {
    const int64_t row = b * block_len + j;
    mj = masked[row] != 0;
    if (mj) {
      Partial p = part[row * n_chunks];
      for (int c = 1; c < n_chunks; ++c) p = merge(p, part[row * n_chunks + c]);
      const float inv = 1.f / p.s;                     // largest probability = 1 / sum exp(x - max)
      cj = inv;
      p2 = (p.m2 > -INFINITY) ? ex2((p.m2 - p.m) * kLog2e) * inv : 0.f;
      aj = p.idx;
    }
    conf[row] = cj;
    argmax[row] = aj;
    if (p2_out) p2_out[row] = p2;
    s_conf[j] = cj;
    s_masked[j] = mj;
    s_score[j] = (mode == SSM_COMMIT_MARGIN) ? cj - p2 : cj;
  }
  __syncthreads();
  bool pass = false;
  if (j < block_len && mj && mode != SSM_COMMIT_TOPK) pass = s_score[j] > threshold;
  if (j < block_len) s_pass[j] = pass;
  if (pass) atomicAdd(&s_npass, 1);
  __syncthreads();
  if (j >= block_len) return;
  bool c = false;
  if (mj) {
    // rank of j among masked positions (confidence descending, position ascending);
    // for threshold/margin only the not-yet-passing ones compete for the min-commit slots
    const bool topk_mode = mode == SSM_COMMIT_TOPK;
    int rank = 0;
    for (int i = 0; i < block_len; ++i) {
      if (!s_masked[i] || i == j) continue;
      if (!topk_mode && s_pass[i]) continue;
      if (s_conf[i] > cj || (s_conf[i] == cj && i < j)) ++rank;
    }
    if (topk_mode) c = rank < topk;
    else c = pass || rank < (min_commit - s_npass);
  }
  commit[b * block_len + j] = c ? 1 : 0;
}

}  // namespace
}  // namespace ssm

namespace {

struct UnmaskPlan {
  int64_t chunk;
  int n_chunks;
  bool vector;
};

UnmaskPlan plan_unmask(int64_t vocab, ssm_dtype dtype, const void* logits) {
  const int esz = dtype == SSM_DTYPE_BF16 ? 2 : 4;
  const int vec = 16 / esz;
  UnmaskPlan p;
  p.vector = ((vocab * esz) % 16 == 0) && (logits == nullptr || ssm::aligned16(logits));
  // both plans cut a row into the same chunks, so the workspace does not depend on the plan
  p.chunk = static_cast<int64_t>(ssm::kUnmaskThreads) * ssm::kUnroll * vec;
  p.n_chunks = static_cast<int>((vocab + p.chunk - 1) / p.chunk);
  return p;
}

}  // namespace

extern "C" {

size_t ssm_unmask_workspace_size(int32_t batch, int32_t block_len, int64_t vocab, ssm_dtype dtype) {
  if (batch <= 0 || block_len <= 0 || vocab <= 0) return 0;
  const UnmaskPlan plan = plan_unmask(vocab, dtype, nullptr);
  return ssm::align_up(static_cast<size_t>(batch) * block_len * plan.n_chunks * sizeof(ssm::Partial), 256);
}

ssm_status ssm_unmask(const void* logits, ssm_dtype dtype, int32_t batch, int32_t block_len,
                      int64_t vocab, const uint8_t* masked, ssm_commit_mode mode, float threshold,
                      int32_t topk, int32_t min_commit, float* conf, int32_t* argmax, float* p2,
                      uint8_t* commit, void* workspace, size_t ws_bytes, ssm_stream_t stream) {
  if (dtype != SSM_DTYPE_BF16 && dtype != SSM_DTYPE_F32) return SSM_ERR_UNSUPPORTED;
  if (batch < 0 || block_len < 0 || vocab <= 0) return SSM_ERR_INVALID_ARG;
  if (mode != SSM_COMMIT_THRESHOLD && mode != SSM_COMMIT_TOPK && mode != SSM_COMMIT_MARGIN)
    return SSM_ERR_INVALID_ARG;
  if (batch == 0 || block_len == 0) return SSM_OK;
  if (block_len > 1024) return SSM_ERR_UNSUPPORTED;
  if (vocab > INT32_MAX) return SSM_ERR_UNSUPPORTED;
  if (!logits || !masked || !conf || !argmax || !commit || !workspace) return SSM_ERR_INVALID_ARG;
  if (mode == SSM_COMMIT_MARGIN && !p2) return SSM_ERR_INVALID_ARG;
  if (topk < 0 || min_commit < 0 || !(threshold == threshold)) return SSM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SSM_ERR_INVALID_ARG;
  if (ws_bytes < ssm_unmask_workspace_size(batch, block_len, vocab, dtype)) return SSM_ERR_CAPACITY;
  const int64_t rows = static_cast<int64_t>(batch) * block_len;
  if (rows > 65535) return SSM_ERR_UNSUPPORTED;
  const UnmaskPlan plan = plan_unmask(vocab, dtype, logits);
  auto* part = static_cast<ssm::Partial*>(workspace);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  dim3 grid(plan.n_chunks, static_cast<unsigned>(rows));
  if (dtype == SSM_DTYPE_BF16) {
    auto* x = static_cast<const __nv_bfloat16*>(logits);
    if (plan.vector)
      ssm::unmask_partial_vec_kernel<__nv_bfloat16, ssm::kUnroll><<<grid, ssm::kUnmaskThreads, 0, st>>>(
          x, vocab, plan.chunk, plan.n_chunks, masked, part);
    else
      ssm::unmask_partial_scalar_kernel<__nv_bfloat16><<<grid, ssm::kUnmaskThreads, 0, st>>>(
          x, vocab, plan.chunk, plan.n_chunks, masked, part);
  } else {
    auto* x = static_cast<const float*>(logits);
    if (plan.vector)
      ssm::unmask_partial_vec_kernel<float, ssm::kUnroll><<<grid, ssm::kUnmaskThreads, 0, st>>>(
          x, vocab, plan.chunk, plan.n_chunks, masked, part);
    else
      ssm::unmask_partial_scalar_kernel<float><<<grid, ssm::kUnmaskThreads, 0, st>>>(
          x, vocab, plan.chunk, plan.n_chunks, masked, part);
  }
  ssm_status s = ssm::launch_status();
  if (s != SSM_OK) return s;
  const int threads = ((block_len + 31) / 32) * 32;
  const size_t shm = static_cast<size_t>(block_len) * (2 * sizeof(float) + 2);
  ssm::unmask_commit_kernel<<<batch, threads, shm, st>>>(block_len, plan.n_chunks, masked, part, mode,
                                                         threshold, topk, min_commit, conf, argmax, p2,
                                                         commit);
  return ssm::launch_status();
}

}  // extern "C"

// ---------------------------------------------------------------------------
// ssm_unmask_noalloc: the same two kernels with their scratch in a fixed,
// statically allocated device array instead of a caller workspace.
// ---------------------------------------------------------------------------

namespace {

// 1 MiB holds 65536 chunk partials: e.g. 512 sequences x 32 positions x 4
// chunks of a 126464-entry bf16 vocabulary.  Every GPU that loads libssm
// keeps this array until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(1) << 20;
static __device__ __align__(256) unsigned char g_unmask_scratch[kNoAllocScratchBytes];

constexpr int kMaxDevices = 64;
std::mutex g_scratch_mu;
void* g_scratch_addr[kMaxDevices] = {};

// Device address of g_unmask_scratch on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up once
// per device (with that device current) and cached.
ssm_status scratch_address(void** out) {
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SSM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return SSM_ERR_UNSUPPORTED;
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (!g_scratch_addr[dev]) {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_unmask_scratch) != cudaSuccess || p == nullptr) return SSM_ERR_CUDA;
    g_scratch_addr[dev] = p;
  }
  *out = g_scratch_addr[dev];
  return SSM_OK;
}

}  // namespace

extern "C" ssm_status ssm_unmask_noalloc(const void* logits, ssm_dtype dtype, int32_t batch, int32_t block_len,
                                         int64_t vocab, const uint8_t* masked, ssm_commit_mode mode,
                                         float threshold, int32_t topk, int32_t min_commit, float* conf,
                                         int32_t* argmax, float* p2, uint8_t* commit, ssm_stream_t stream) {
  if (batch > 0 && block_len > 0 && vocab > 0 &&
      ssm_unmask_workspace_size(batch, block_len, vocab, dtype) > kNoAllocScratchBytes)
    return SSM_ERR_CAPACITY;
  void* scratch = nullptr;
  const ssm_status s = scratch_address(&scratch);
  if (s != SSM_OK) return s;
  // The chunk partials are written before they are read on every call, so the
  // previous call's contents never need clearing.
  return ssm_unmask(logits, dtype, batch, block_len, vocab, masked, mode, threshold, topk, min_commit, conf,
                    argmax, p2, commit, scratch, kNoAllocScratchBytes, stream);
}
