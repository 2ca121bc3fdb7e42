// unmask.cu -- confidence-based unmasking (Sec. 4.2 "Baselines": Vanilla top-1
// and parallel threshold decoding; Sec. 4.6: margin decoding), and
// ssm_unmask_topk, which also enqueues the retained suffix positions' top-k
// (topk.cu) for the next step's Eq. 6.
//
// Pass 1 (unmask_stream_kernel): the masked rows of logits are cut into 16 KB
// stages, numbered row-major over the call, and every persistent CTA (three per
// SM, one wave) takes one contiguous range of the same number of stages, so the
// CTAs finish together whatever the row length and batch.  Each thread streams
// its own 64-byte slices of successive stages from HBM into a private two-stage
// shared-memory ring with 16-byte cp.async copies, so the read runs ahead of the
// arithmetic without any barrier (a thread only reads back what it copied
// itself), and folds every stage into a running (max, first argmax, sum of
// exp(x - max)) plus, when p2 is wanted, the second-largest value.  Where its
// range leaves a row (or ends), the CTA merges its 256 running states into one
// partial of that row.  Rows whose length or alignment rules out 16-byte copies
// take unmask_partial_scalar_kernel on the same ranges.
// Pass 2 (unmask_commit_kernel): one CTA per batch row merges the partials of
// its positions (one per CTA whose range meets the row), writes conf / argmax /
// p2 and applies the commit rule.  Logits of unmasked rows are never read.
#include <cuda_bf16.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "common.cuh"
#include "sm100_ptx.cuh"
#include "stream.cuh"
#include "topk.cuh"

namespace ssm {
namespace {

constexpr int kUnmaskThreads = 256;
constexpr int kMaxStreamCtas = 768;                // grid cap of the streaming pass (three CTAs per SM, <= 256 SMs)
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
  __device__ static void unpack(const uint4& v, float (&f)[4]) {
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
  }
  __device__ static float scalar(const float* p, int64_t i) { return p[i]; }
};

// ---------------------------------------------------------------------------
// Streaming pass: bulk copies into a shared-memory ring, 8 consumer warps
// ---------------------------------------------------------------------------

constexpr int kStreamThreads = 256;
constexpr int kStageBytes = 16384;                     // one stage: 64 bytes per thread
constexpr int kStreamStages = 2;                       // stages in flight per thread
constexpr int kVecPerThread = kStageBytes / 16 / kStreamThreads;  // 4


// Running per-thread state over one row's stages in a CTA range: max m1 (first index idx), second
// largest m2 (a repeated maximum counts twice) and s = sum exp(x - m1).
struct RunState {
  float m1, m2, s;
  int idx;
};

// (three CTAs per SM: the grid is one wave of them)
template <typename T, bool NEED_SECOND>
__global__ void __launch_bounds__(kStreamThreads, 3) unmask_stream_kernel(
    const T* __restrict__ logits, int64_t vocab, int32_t n_stage, int64_t per, int64_t n_total, int kr,
    const uint8_t* __restrict__ masked, Partial* __restrict__ part) {
  pdl_enter();
  constexpr int ESZ = sizeof(T);
  extern __shared__ uint8_t smem_raw[];
  uint8_t* ring = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 127) & ~uintptr_t(127));
  // each thread's copy of its 64 bytes of the stage that holds its running maximum
  uint4* keep = reinterpret_cast<uint4*>(ring + kStreamStages * kStageBytes) + threadIdx.x * kVecPerThread;
  __shared__ Partial wpart[kStreamThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  constexpr int64_t SE = kStageBytes / ESZ;  // elements per stage
  // this CTA's stages [g0, g1)
  const int64_t g0 = static_cast<int64_t>(blockIdx.x) * per;
  const int64_t g1 = min(n_total, g0 + per);
  // issue side runs kStreamStages stages ahead of the compute side; a thread only ever
  // reads the shared-memory bytes it copied itself, so no barrier is needed between them
  StageCursor is = stage_begin<T>(g0, g1, n_stage, SE, vocab, masked);
  auto issue = [&](int slot) {
    if (is.g < g1) {
      const uint8_t* src = reinterpret_cast<const uint8_t*>(logits + is.row * vocab + is.e0);
      uint8_t* dst = ring + slot * kStageBytes;
#pragma unroll
      for (int u = 0; u < kVecPerThread; ++u) {
        const int vi = u * kStreamThreads + threadIdx.x;
        if (vi * 16 < is.bytes) cp_async16(dst + vi * 16, src + vi * 16);
      }
      stage_next<T>(is, g1, n_stage, SE, vocab, masked);
    }
    cp_async_commit();
  };
#pragma unroll
  for (int k = 0; k < kStreamStages; ++k) issue(k);

  StageCursor cs = stage_begin<T>(g0, g1, n_stage, SE, vocab, masked);
  // this CTA's slot among the CTAs whose ranges meet a row: 0 for every row but the first
  const int64_t first_row = g0 / n_stage;
  const int first_slot = static_cast<int>(blockIdx.x - (first_row * n_stage) / per);
  int slot = 0;
  while (cs.g < g1) {
    const int64_t row = cs.row;
    RunState r{-INFINITY, -INFINITY, 0.f, INT_MAX};
    while (cs.g < g1 && cs.row == row) {
      cp_async_wait<kStreamStages - 1>();
      const int stage_bytes = cs.bytes;
      const uint4* sv = reinterpret_cast<const uint4*>(ring + slot * kStageBytes);
      uint4 v[kVecPerThread];
      bool in[kVecPerThread];
      const uint32_t ninf = (ESZ == 2) ? 0xFF80FF80u : 0xFF800000u;
#pragma unroll
      for (int u = 0; u < kVecPerThread; ++u) {
        const int vi = u * kStreamThreads + threadIdx.x;
        in[u] = vi * 16 < stage_bytes;
        v[u] = in[u] ? sv[vi] : make_uint4(ninf, ninf, ninf, ninf);
      }
      const int64_t base = cs.e0;
      // this thread's values of the stage as fp32 (entries past a short last stage are -inf)
      constexpr int PER = kVecPerThread * 16 / ESZ;  // 32 bf16 or 16 fp32 values
      float f[PER];
#pragma unroll
      for (int u = 0; u < kVecPerThread; ++u) {
        const uint32_t w4[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
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
      // stage maximum (four chains of 3-input max) and, when asked for, the second largest
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
      const float cm1 = fmaxf(fmaxf(c4[0], c4[1]), fmaxf(c4[2], c4[3]));
      // The argmax (first position of the maximum) and, when wanted, the second largest (a
      // repeated maximum counts twice) are taken once, where the range leaves the row, from a
      // copy of the maximum's stage: a stage that raises a lane's maximum only stores its 64
      // bytes (four 16-byte shared-memory stores; on most stages some lane of the warp does).
      // The second largest is then the larger of the second largest inside that stage and the
      // largest value of every other stage, which r.m2 keeps.
      if (cm1 > r.m1) {
        if constexpr (NEED_SECOND) r.m2 = fmaxf(r.m2, r.m1);
#pragma unroll
        for (int u = 0; u < kVecPerThread; ++u) keep[u] = v[u];
        r.idx = static_cast<int>(base);   // the kept stage's first entry
        if (r.m1 > -INFINITY) r.s *= ex2((r.m1 - cm1) * kLog2e);
        r.m1 = cm1;
      } else if constexpr (NEED_SECOND) {
        r.m2 = fmaxf(r.m2, cm1);
      }
      if (r.m1 > -INFINITY) {
        const float mb = r.m1 * kLog2e;
        float sa[4] = {0.f, 0.f, 0.f, 0.f}, sb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int e = 0; e < PER; e += 2) {
          float t0, t1;
          ffma2(t0, t1, f[e], f[e + 1], kLog2e, kLog2e, -mb, -mb);
          fadd2_acc(sa[(e >> 1) & 3], sb[(e >> 1) & 3], ex2(t0), ex2(t1));
        }
        r.s += ((sa[0] + sb[0]) + (sa[1] + sb[1])) + ((sa[2] + sb[2]) + (sa[3] + sb[3]));
      }
      // the slot has been read and used: refill it with the stage kStreamStages ahead
      issue(slot);
      slot = (slot + 1) % kStreamStages;
      stage_next<T>(cs, g1, n_stage, SE, vocab, masked);
    }
    // the CTA's partial of the row: per-warp shuffles, then thread 0 merges the eight
    // the kept stage: first position of the maximum and, when wanted, its second largest
    if (r.m1 > -INFINITY) {
      const int tbase = r.idx + static_cast<int>(threadIdx.x) * (16 / ESZ);
      constexpr int EPV = 16 / ESZ;
      int best = INT_MAX;
      float s2 = -INFINITY, m1l = -INFINITY;
#pragma unroll
      for (int u = kVecPerThread - 1; u >= 0; --u) {
        const uint4 kv = keep[u];
        const uint32_t w4[4] = {kv.x, kv.y, kv.z, kv.w};
#pragma unroll
        for (int e = EPV - 1; e >= 0; --e) {
          const float f = (ESZ == 2) ? ((e & 1) ? hi_bf16(w4[e >> 1]) : lo_bf16(w4[e >> 1])) : __uint_as_float(w4[e]);
          best = (f == r.m1) ? tbase + u * kStreamThreads * EPV + e : best;
          if constexpr (NEED_SECOND) {
            s2 = fmaxf(s2, fminf(m1l, f));
            m1l = fmaxf(m1l, f);
          }
        }
      }
      r.idx = best;
      if constexpr (NEED_SECOND) r.m2 = fmaxf(r.m2, s2);
    }
    Partial pw{r.m1, r.s, r.idx, r.m2};
#pragma unroll
    for (int d = 16; d >= 1; d >>= 1) pw = merge(pw, shfl_partial(pw, d));
    if (lane == 0) wpart[warp] = pw;
    __syncthreads();
    if (threadIdx.x == 0) {
      Partial q = wpart[0];
      for (int w2 = 1; w2 < kStreamThreads / 32; ++w2) q = merge(q, wpart[w2]);
      // slot of this CTA among the CTAs whose ranges meet the row
      part[row * kr + (row == first_row ? first_slot : 0)] = q;
    }
    __syncthreads();
  }
  cp_async_wait<0>();
}

// Rows whose length or alignment rules out 16-byte vectors: the same stage ranges,
// one element per thread per step, online (max, second, first index) then the exp sum,
// for each row the range meets.
template <typename T>
__global__ void __launch_bounds__(kUnmaskThreads) unmask_partial_scalar_kernel(
    const T* __restrict__ logits, int64_t vocab, int32_t n_stage, int64_t per, int64_t n_total, int kr,
    const uint8_t* __restrict__ masked, Partial* __restrict__ part) {
  pdl_enter();
  constexpr int64_t SE = kStageBytes / static_cast<int64_t>(sizeof(T));
  __shared__ Partial sp[kUnmaskThreads / 32];
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int64_t g0 = static_cast<int64_t>(blockIdx.x) * per;
  const int64_t g1 = min(n_total, g0 + per);
  for (int64_t g = g0; g < g1;) {
    const int64_t row = g / n_stage;
    const int64_t gr = min(g1, (row + 1) * n_stage);   // this row's stages in the range end here
    if (masked[row]) {
      const int64_t c0 = (g - row * n_stage) * SE;
      const int64_t c1 = min(vocab, (gr - row * n_stage) * SE);
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
      if (lane == 0) sp[warp] = p;
      __syncthreads();
      if (warp == 0) {
        p = (lane < kUnmaskThreads / 32) ? sp[lane] : Partial{-INFINITY, 0.f, INT_MAX, -INFINITY};
#pragma unroll
        for (int d = 4; d >= 1; d >>= 1) p = merge(p, shfl_partial(p, d));
        if (lane == 0) part[row * kr + (static_cast<int64_t>(blockIdx.x) - (row * n_stage) / per)] = p;
      }
      __syncthreads();
    }
    g = gr;
  }
}

// One CTA per batch row; thread j owns block position j.
__global__ void __launch_bounds__(1024) unmask_commit_kernel(
    int block_len, int32_t n_stage, int64_t per, int kr, const uint8_t* __restrict__ masked,
    const Partial* __restrict__ part,
    int mode, float threshold, int topk, int min_commit, float* __restrict__ conf,
    int32_t* __restrict__ argmax, float* __restrict__ p2_out, uint8_t* __restrict__ commit) {
  pdl_enter();
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
    // the row's partials (one per CTA whose stage range meets the row) are loaded eight at a
    // time, independently, then merged (a chain of dependent loads would cost one memory
    // latency per partial), and they are loaded together with the row's mask byte: an
    // unmasked row's slots hold no partial of this call, and what they hold is not used
    const int n_part = static_cast<int>((row * n_stage + n_stage - 1) / per - (row * n_stage) / per + 1);
    const Partial* pr = part + row * kr;
    Partial p = pr[0];
    mj = masked[row] != 0;
    for (int c0 = 1; c0 < n_part; c0 += 8) {
      Partial q[8];
#pragma unroll
      for (int c = 0; c < 8; ++c) q[c] = pr[min(c0 + c, n_part - 1)];
#pragma unroll
      for (int c = 0; c < 8; ++c)
        if (c0 + c < n_part) p = merge(p, q[c]);
    }
    if (mj) {
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
  int32_t n_stage;  // 16 KB stages per row
  int64_t per;      // stages per CTA
  int64_t total;    // stages of the call (rows x n_stage)
  int grid;         // CTAs
  int kr;           // partial slots per row: at most this many CTA ranges meet a row
  bool vector;
};

// Every CTA takes `per` consecutive stages of the call, per = ceil(total / CTAs) with at
// most max_ctas CTAs; a row's n_stage stages then meet at most ceil((n_stage - 1) / per) + 1
// ranges (and never more than n_stage).  Fewer CTAs give longer ranges and fewer slots per
// row, so the workspace is sized at the grid cap and fits every grid at or below it.
UnmaskPlan plan_unmask(int64_t rows, int64_t vocab, ssm_dtype dtype, const void* logits, int max_ctas) {
  const int esz = dtype == SSM_DTYPE_BF16 ? 2 : 4;
  UnmaskPlan p;
  p.vector = ((vocab * esz) % 16 == 0) && (logits == nullptr || ssm::aligned16(logits));
  const int64_t stage_elems = ssm::kStageBytes / esz;
  p.n_stage = static_cast<int32_t>((vocab + stage_elems - 1) / stage_elems);
  p.total = rows * p.n_stage;
  const int64_t g = std::max<int64_t>(1, std::min<int64_t>(max_ctas, p.total));
  p.per = (p.total + g - 1) / g;
  p.grid = static_cast<int>((p.total + p.per - 1) / p.per);
  p.kr = static_cast<int>(std::min<int64_t>(p.n_stage, (p.n_stage - 1 + p.per - 1) / p.per + 1));
  return p;
}

// The ring exceeds the default 48 KB of dynamic shared memory: opt in once per device
// and kernel (one static flag per instantiation of this function, i.e. per kernel).
template <auto kernel>
bool stream_attr_set(size_t bytes) {
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

// One streaming launch: the kernel form for the dtype and p2 tracking.  The ring (two 16 KB
// stages) and a 64-byte copy per thread of its maximum's stage (16 KB) exceed the default
// 48 KB of dynamic shared memory.
template <typename T, bool NEED_SECOND>
ssm_status launch_stream_form(int grid, cudaStream_t st, const T* x, int64_t vocab, const UnmaskPlan& plan,
                              const uint8_t* masked, ssm::Partial* part) {
  const size_t smem = (ssm::kStreamStages + 1) * ssm::kStageBytes + 128;
  if (!stream_attr_set<ssm::unmask_stream_kernel<T, NEED_SECOND>>(smem)) return SSM_ERR_CUDA;
  ssm::launch_k(ssm::unmask_stream_kernel<T, NEED_SECOND>, dim3(grid), dim3(ssm::kStreamThreads), smem, st, x, vocab,
                plan.n_stage, plan.per, plan.total, plan.kr, masked, part);
  return SSM_OK;
}

template <typename T>
ssm_status launch_stream(const T* x, bool need_second, int grid, cudaStream_t st, int64_t vocab,
                         const UnmaskPlan& plan, const uint8_t* masked, ssm::Partial* part) {
  return need_second ? launch_stream_form<T, true>(grid, st, x, vocab, plan, masked, part)
                     : launch_stream_form<T, false>(grid, st, x, vocab, plan, masked, part);
}

}  // namespace

extern "C" {

size_t ssm_unmask_workspace_size(int32_t batch, int32_t block_len, int64_t vocab, ssm_dtype dtype) {
  if (batch <= 0 || block_len <= 0 || vocab <= 0) return 0;
  const UnmaskPlan plan =
      plan_unmask(static_cast<int64_t>(batch) * block_len, vocab, dtype, nullptr, ssm::kMaxStreamCtas);
  return ssm::align_up(static_cast<size_t>(batch) * block_len * plan.kr * sizeof(ssm::Partial), 256);
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
  // one wave: three CTAs per SM are resident (registers)
  const UnmaskPlan plan =
      plan_unmask(rows, vocab, dtype, logits, std::min(3 * ssm::num_sms(), ssm::kMaxStreamCtas));
  auto* part = static_cast<ssm::Partial*>(workspace);
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  const int stream_grid = plan.grid;
  const bool need_second = p2 != nullptr || mode == SSM_COMMIT_MARGIN;
  if (plan.vector) {
    const ssm_status s0 = dtype == SSM_DTYPE_BF16
        ? launch_stream(static_cast<const __nv_bfloat16*>(logits), need_second, stream_grid, st, vocab, plan, masked,
                        part)
        : launch_stream(static_cast<const float*>(logits), need_second, stream_grid, st, vocab, plan, masked, part);
    if (s0 != SSM_OK) return s0;
  } else if (dtype == SSM_DTYPE_BF16) {
    ssm::launch_k(ssm::unmask_partial_scalar_kernel<__nv_bfloat16>, dim3(stream_grid), dim3(ssm::kUnmaskThreads), 0,
                  st, static_cast<const __nv_bfloat16*>(logits), vocab, plan.n_stage, plan.per, plan.total, plan.kr,
                  masked, part);
  } else {
    ssm::launch_k(ssm::unmask_partial_scalar_kernel<float>, dim3(stream_grid), dim3(ssm::kUnmaskThreads), 0, st,
                  static_cast<const float*>(logits), vocab, plan.n_stage, plan.per, plan.total, plan.kr, masked, part);
  }
  ssm_status s = ssm::launch_status();
  if (s != SSM_OK) return s;
  const int threads = ((block_len + 31) / 32) * 32;
  const size_t shm = static_cast<size_t>(block_len) * (2 * sizeof(float) + 2);
  // The commit kernel is launched with programmatic dependent launch also when the stream is
  // being captured (a programmatic edge in the graph): its few small CTAs fit beside the stream
  // kernel's, so its launch and CTA start overlap the stream kernel's tail; its griddepcontrol
  // wait still orders every read after the stream kernel's partials.
  ssm::launch_k_pdl(ssm::unmask_commit_kernel, dim3(batch), dim3(threads), shm, st, block_len, plan.n_stage,
                    plan.per, plan.kr, masked, static_cast<const ssm::Partial*>(part), static_cast<int>(mode),
                    threshold, topk, min_commit, conf, argmax, p2, commit);
  return ssm::launch_status();
}

ssm_status ssm_unmask_topk(const void* logits, ssm_dtype dtype, int32_t batch, int32_t block_len, int64_t vocab,
                           const uint8_t* masked, ssm_commit_mode mode, float threshold, int32_t topk,
                           int32_t min_commit, float* conf, int32_t* argmax, float* p2, uint8_t* commit,
                           const void* suffix_logits, int64_t n_suffix_rows, int32_t k, int32_t* ids,
                           float* probs, void* workspace, size_t ws_bytes, ssm_stream_t stream) {
  if (n_suffix_rows < 0) return SSM_ERR_INVALID_ARG;
  if (n_suffix_rows == 0)
    return ssm_unmask(logits, dtype, batch, block_len, vocab, masked, mode, threshold, topk, min_commit, conf,
                      argmax, p2, commit, workspace, ws_bytes, stream);
  if (dtype != SSM_DTYPE_BF16 && dtype != SSM_DTYPE_F32) return SSM_ERR_UNSUPPORTED;
  if (k < 1 || k > 8) return SSM_ERR_UNSUPPORTED;
  if (vocab <= 0 || k > vocab || !suffix_logits || !ids || !probs) return SSM_ERR_INVALID_ARG;
  if (batch < 0 || block_len < 0) return SSM_ERR_INVALID_ARG;
  if (batch == 0 || block_len == 0)
    return ssm_suffix_topk(suffix_logits, dtype, n_suffix_rows, vocab, k, ids, probs, stream);
  if (mode != SSM_COMMIT_THRESHOLD && mode != SSM_COMMIT_TOPK && mode != SSM_COMMIT_MARGIN)
    return SSM_ERR_INVALID_ARG;
  if (block_len > 1024 || vocab > INT32_MAX) return SSM_ERR_UNSUPPORTED;
  if (!logits || !masked || !conf || !argmax || !commit || !workspace) return SSM_ERR_INVALID_ARG;
  if (mode == SSM_COMMIT_MARGIN && !p2) return SSM_ERR_INVALID_ARG;
  if (topk < 0 || min_commit < 0 || !(threshold == threshold)) return SSM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SSM_ERR_INVALID_ARG;
  if (ws_bytes < ssm_unmask_workspace_size(batch, block_len, vocab, dtype)) return SSM_ERR_CAPACITY;
  const int64_t rows = static_cast<int64_t>(batch) * block_len;
  if (rows > 65535) return SSM_ERR_UNSUPPORTED;
  // the top-k pass's own conditions, checked first so that an error enqueues nothing
  const int esz = dtype == SSM_DTYPE_BF16 ? 2 : 4;
  if (!ssm::aligned16(suffix_logits) || (vocab * esz) % 16 != 0) return SSM_ERR_UNSUPPORTED;
  const int64_t nchunk = (vocab * esz + ssm::topk::kTopStageBytes - 1) / ssm::topk::kTopStageBytes;
  if (ssm::topk::kTopStages * ssm::topk::kTopStageBytes + nchunk * ssm::topk::kTopThreads * esz + 128 >
      ssm::topk::kTopMaxSmem)
    return SSM_ERR_UNSUPPORTED;
  // The two streaming passes back to back on the stream: the block rows' unmasking (its stream
  // and commit kernels) and the suffix rows' top-k.  A single kernel serving both kinds of
  // rows was measured slower than the two (it holds fewer bytes in flight per SM than the
  // top-k pass alone), so the call enqueues the faster pair.
  const ssm_status s = ssm_unmask(logits, dtype, batch, block_len, vocab, masked, mode, threshold, topk, min_commit,
                                  conf, argmax, p2, commit, workspace, ws_bytes, stream);
  if (s != SSM_OK) return s;
  return ssm_suffix_topk(suffix_logits, dtype, n_suffix_rows, vocab, k, ids, probs, stream);
}

}  // extern "C"

// ---------------------------------------------------------------------------
// ssm_unmask_noalloc: the same two kernels with their scratch in a fixed,
// statically allocated device array instead of a caller workspace.
// ---------------------------------------------------------------------------

namespace {

// 2 MiB holds 131072 16-byte row partials: two per row for every call of up to
// 65535 positions of a 126464-entry bf16 or fp32 vocabulary (more per row only
// for calls with fewer rows than the streaming pass has CTAs).  Every GPU that
// loads libssm keeps this array until the process exits.
constexpr size_t kNoAllocScratchBytes = size_t(2) << 20;
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
  // The row partials are written before they are read on every call, so the
  // previous call's contents never need clearing.
  return ssm_unmask(logits, dtype, batch, block_len, vocab, masked, mode, threshold, topk, min_commit, conf,
                    argmax, p2, commit, scratch, kNoAllocScratchBytes, stream);
}
