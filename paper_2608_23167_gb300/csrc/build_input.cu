// build_input.cu -- sparse step input with soft suffix embeddings
// (Sec. 3.2 "Soft Suffix Embedding Mixing", Eqs. 6-8, and "Sparse Input
// Construction": X~_t = [P; B_t; R_t] keeping the original positions).
//
// One CTA per output row.  Prompt and block rows are embedding-row copies;
// a retained suffix row reads the [MASK] row plus its k previous-step
// candidate rows and writes (1-alpha) e_mask + alpha * sum_j p~_j e_j.  Every
// access is a 16-byte vector (8 bf16 values), so a row of hidden 4096 is 512
// coalesced vectors.  The work is a gather: HBM-bound, no tensor cores.
#include <cuda_bf16.h>

#include "common.cuh"
#include "suffix_geom.cuh"

namespace ssm {
namespace {

constexpr int kBuildThreads = 128;
constexpr int kMaxK = 32;

struct BuildParams {
  const ssm_step_problem* problems;  // null: uniform batch
  int32_t n_problems;
  // uniform description (problems == null)
  int32_t u_n_prefix, u_n_suffix, u_block_start;
  int32_t block_len;
  const int32_t* block_tokens;
  const int32_t* prefix_tokens;
  const int32_t* suffix_pos;
  const ssm_suffix_cfg* cfgs;  // per problem: the selection, made here (suffix_pos unused), or null
  int32_t* suffix_pos_out;     // with cfgs: R_t of every problem written here too (may be null)
  const uint4* embed;        // [vocab, hidden/8] 16-byte vectors
  int64_t vocab;
  int32_t hvec;              // hidden / 8
  int32_t mask_id;
  const int32_t* topk_ids;
  const float* topk_prob;
  int32_t k;
  float alpha;
  uint4* x_out;
  int32_t* pos_out;
  unsigned* err;
};

__device__ __forceinline__ void unpack8(const uint4& v, float (&f)[8]) {
  const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
  for (int i = 0; i < 4; ++i) {
    f[2 * i] = __uint_as_float(w[i] << 16);
    f[2 * i + 1] = __uint_as_float(w[i] & 0xFFFF0000u);
  }
}

__device__ __forceinline__ uint32_t pack2(float a, float b) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// A row copy with every thread's loads issued before its stores (four 16-byte vectors per
// thread in flight, not one load-store round trip per vector).
__device__ __forceinline__ void copy_row(const uint4* __restrict__ src, uint4* __restrict__ dst, int hvec) {
  constexpr int U = 4;
  for (int v0 = threadIdx.x; v0 < hvec; v0 += U * kBuildThreads) {
    uint4 t[U];
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (v0 + u * kBuildThreads < hvec) t[u] = __ldg(src + v0 + u * kBuildThreads);
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (v0 + u * kBuildThreads < hvec) dst[v0 + u * kBuildThreads] = t[u];
  }
}

__device__ __forceinline__ void zero_row(uint4* __restrict__ dst, int hvec) {
  for (int v = threadIdx.x; v < hvec; v += kBuildThreads) dst[v] = make_uint4(0, 0, 0, 0);
}

// COLS: 16-byte columns of a retained suffix row each thread gathers per pass, with every load
// of the pass in flight (one pass of the row per COLS * kBuildThreads columns).  Two columns
// halve a hidden-4096 row's memory round trips but take 88 registers against 52 (five CTAs
// per SM instead of nine): the host takes them for small launches (two_columns below).
template <int COLS>
__global__ void __launch_bounds__(kBuildThreads) build_step_input_kernel(const BuildParams p) {
  pdl_enter();
  __shared__ int32_t s_ids[kMaxK];
  __shared__ float s_w[kMaxK];
  __shared__ int32_t s_n;
  __shared__ int32_t s_bad;
  __shared__ int32_t s_mismatch;

  const int prob = blockIdx.y;
  const int r = blockIdx.x;
  int64_t block_tok_off, prefix_tok_off, suffix_off, out_row;
  int32_t n_prefix, n_suffix, block_start;
  if (p.problems) {
    const ssm_step_problem q = p.problems[prob];
    block_tok_off = q.block_tok_off;
    prefix_tok_off = q.prefix_tok_off;
    suffix_off = q.suffix_off;
    out_row = q.out_row;
    n_prefix = q.n_prefix;
    n_suffix = q.n_suffix;
    block_start = q.block_start;
  } else {
    n_prefix = p.u_n_prefix;
    n_suffix = p.u_n_suffix;
    block_start = p.u_block_start;
    block_tok_off = static_cast<int64_t>(prob) * p.block_len;
    prefix_tok_off = static_cast<int64_t>(prob) * n_prefix;
    suffix_off = 0;  // positions shared by the batch; top-k rows indexed below
    out_row = static_cast<int64_t>(prob) * (n_prefix + p.block_len + n_suffix);
  }
  const int32_t rows = n_prefix + p.block_len + n_suffix;
  if (r >= rows) return;
  uint4* dst = p.x_out + (out_row + r) * p.hvec;

  // original position id of this row (Sec. 3.2: retained tokens keep their positions); with
  // per-problem selections a retained suffix row's position is its rank in R_t mapped to the
  // position in closed form (Eqs. 2-5, below), so no separate selection pass is needed
  if (threadIdx.x == 0 && (p.problems || prob == 0) && !(p.cfgs && r >= n_prefix + p.block_len)) {
    int32_t pos;
    if (r < n_prefix) pos = r;
    else if (r < n_prefix + p.block_len) pos = block_start + (r - n_prefix);
    else pos = p.suffix_pos[suffix_off + (r - n_prefix - p.block_len)];
    if (p.pos_out) p.pos_out[(p.problems ? out_row : 0) + r] = pos;
  }

  if (r < n_prefix + p.block_len) {
    const int32_t tok = (r < n_prefix) ? p.prefix_tokens[prefix_tok_off + r]
                                       : p.block_tokens[block_tok_off + (r - n_prefix)];
    if (tok < 0 || tok >= p.vocab) {
      if (threadIdx.x == 0) record_error(p.err, SSM_ERR_DEVICE_INPUT);
      zero_row(dst, p.hvec);
      return;
    }
    copy_row(p.embed + static_cast<int64_t>(tok) * p.hvec, dst, p.hvec);
    return;
  }

  // retained suffix row i: Eq. 6 renormalisation, Eq. 7 soft embedding, Eq. 8 mix
  const int64_t i = r - n_prefix - p.block_len;
  const int64_t cand = p.problems ? (suffix_off + i) * p.k
                                  : (static_cast<int64_t>(prob) * n_suffix + i) * p.k;
  if (p.cfgs && threadIdx.x == 32) {
    // this row's position, its rank i in R_t mapped in closed form, by a second warp while the
    // first one gathers the candidates
    const SuffixGeom g = make_geom(p.cfgs[prob]);
    int32_t nl, nm, nt;
    region_counts(g, nl, nm, nt);
    if (nl + nm + nt != n_suffix) {   // the problem table disagrees with its selection
      s_mismatch = 1;
      record_error(p.err, SSM_ERR_DEVICE_INPUT);
    } else {
      s_mismatch = 0;
      const int32_t pos = static_cast<int32_t>(retained_position(g, nl, nm, i));
      if (p.pos_out) p.pos_out[out_row + r] = pos;
      if (p.suffix_pos_out) p.suffix_pos_out[suffix_off + i] = pos;
    }
  }
  if (threadIdx.x < 32) {
    // the k candidates (id, p) of the previous step, lane j loading candidate j (k <= 32), so
    // that their loads are in flight together; an id of -1 is absent, an id outside the
    // vocabulary is an input error
    const int lane = threadIdx.x;
    const bool have = p.topk_ids != nullptr && lane < p.k;
    const int32_t id = have ? p.topk_ids[cand + lane] : -1;
    const float pj = have ? p.topk_prob[cand + lane] : 0.f;
    const bool bad = id != -1 && (id < 0 || id >= p.vocab);
    const unsigned use = __ballot_sync(0xffffffffu, id != -1 && !bad);
    const unsigned badm = __ballot_sync(0xffffffffu, bad);
    // the renormaliser sum(p) over the kept candidates, added in candidate order
    float z = 0.f;
    for (int j = 0; j < p.k; ++j) {
      const float w = __shfl_sync(0xffffffffu, pj, j);
      if ((use >> j) & 1u) z += w;
    }
    const int n = (z > 0.f) ? __popc(use) : 0;   // no prediction: the row keeps e_mask
    const float scale = n ? p.alpha / z : 0.f;   // alpha * p_j / sum(p) = alpha * p~_j
    if (n && ((use >> lane) & 1u)) {
      const int slot = __popc(use & ((1u << lane) - 1u));
      s_ids[slot] = id;
      s_w[slot] = pj * scale;
    }
    if (lane == 0) {
      s_n = n;
      s_bad = badm != 0u;
      if (badm) record_error(p.err, SSM_ERR_DEVICE_INPUT);
    }
  }
  __syncthreads();
  if (s_bad || (p.cfgs && s_mismatch)) {
    zero_row(dst, p.hvec);
    return;
  }
  const int n = s_n;
  const uint4* e_mask = p.embed + static_cast<int64_t>(p.mask_id) * p.hvec;
  if (n == 0) {
    copy_row(e_mask, dst, p.hvec);
    return;
  }
  const float keep = 1.f - p.alpha;
  // gather the candidate rows six at a time: all of a chunk's loads (and the [MASK] row's) for
  // the pass's COLS columns are in flight together; the products are added in candidate order
  constexpr int C = 6;
  if constexpr (COLS == 1) {
    for (int v = threadIdx.x; v < p.hvec; v += kBuildThreads) {
      float acc[8];
      const uint4 mv = __ldg(e_mask + v);
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[c] = 0.f;
      for (int j = 0; j < n; j += C) {
        uint4 ev[C];
#pragma unroll
        for (int u = 0; u < C; ++u)
          if (j + u < n) ev[u] = __ldg(p.embed + static_cast<int64_t>(s_ids[j + u]) * p.hvec + v);
#pragma unroll
        for (int u = 0; u < C; ++u) {
          if (j + u < n) {
            float f[8];
            unpack8(ev[u], f);
            const float w = s_w[j + u];
#pragma unroll
            for (int c = 0; c < 8; ++c) acc[c] = fmaf(w, f[c], acc[c]);
          }
        }
      }
      float m[8];
      unpack8(mv, m);
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[c] = fmaf(keep, m[c], acc[c]);
      uint4 o;
      o.x = pack2(acc[0], acc[1]);
      o.y = pack2(acc[2], acc[3]);
      o.z = pack2(acc[4], acc[5]);
      o.w = pack2(acc[6], acc[7]);
      dst[v] = o;
    }
    return;
  }
  for (int v0 = threadIdx.x; v0 < p.hvec; v0 += COLS * kBuildThreads) {
    bool on[COLS];
    float acc[COLS][8];
    uint4 mv[COLS];
#pragma unroll
    for (int q = 0; q < COLS; ++q) {
      on[q] = v0 + q * kBuildThreads < p.hvec;
      mv[q] = on[q] ? __ldg(e_mask + v0 + q * kBuildThreads) : make_uint4(0, 0, 0, 0);
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[q][c] = 0.f;
    }
    for (int j = 0; j < n; j += C) {
      uint4 ev[COLS][C];
#pragma unroll
      for (int u = 0; u < C; ++u) {
        if (j + u < n) {
          const uint4* rowp = p.embed + static_cast<int64_t>(s_ids[j + u]) * p.hvec + v0;
#pragma unroll
          for (int q = 0; q < COLS; ++q)
            if (on[q]) ev[q][u] = __ldg(rowp + q * kBuildThreads);
        }
      }
#pragma unroll
      for (int u = 0; u < C; ++u) {
        if (j + u < n) {
          const float w = s_w[j + u];
#pragma unroll
          for (int q = 0; q < COLS; ++q) {
            if (on[q]) {
              float f[8];
              unpack8(ev[q][u], f);
#pragma unroll
              for (int c = 0; c < 8; ++c) acc[q][c] = fmaf(w, f[c], acc[q][c]);
            }
          }
        }
      }
    }
#pragma unroll
    for (int q = 0; q < COLS; ++q) {
      if (!on[q]) continue;
      float m[8];
      unpack8(mv[q], m);
#pragma unroll
      for (int c = 0; c < 8; ++c) acc[q][c] = fmaf(keep, m[c], acc[q][c]);
      uint4 o;
      o.x = pack2(acc[q][0], acc[q][1]);
      o.y = pack2(acc[q][2], acc[q][3]);
      o.z = pack2(acc[q][4], acc[q][5]);
      o.w = pack2(acc[q][6], acc[q][7]);
      dst[v0 + q * kBuildThreads] = o;
    }
  }
}

// Small launches take the two-column form: up to about one and a half waves of it (five CTAs per
// SM at its 88 registers; the serving batch's 808 rows measured 1 us faster with it), where the
// row's round trips, not the bytes in flight, set the time.  Large launches (the sweep's
// 11008 CTAs) keep nine CTAs per SM of the one-column form.
inline bool two_columns(int64_t ctas) { return ctas <= 8ll * num_sms(); }

ssm_status check_common(const void* embed, int64_t vocab, int32_t hidden, int32_t mask_id, int32_t k,
                        float alpha, int32_t block_len, const void* x_out) {
  if (!embed || !x_out || vocab <= 0 || hidden <= 0 || block_len < 0) return SSM_ERR_INVALID_ARG;
  if (hidden % 8 != 0) return SSM_ERR_UNSUPPORTED;
  if (!aligned16(embed) || !aligned16(x_out)) return SSM_ERR_INVALID_ARG;
  if (mask_id < 0 || mask_id >= vocab) return SSM_ERR_INVALID_ARG;
  if (k < 0 || k > kMaxK) return SSM_ERR_UNSUPPORTED;
  if (!(alpha >= 0.f && alpha <= 1.f)) return SSM_ERR_INVALID_ARG;
  return SSM_OK;
}

}  // namespace
}  // namespace ssm

extern "C" {

ssm_status ssm_build_step_input(const int32_t* block_tokens, const int32_t* prefix_tokens,
                                int32_t batch, int32_t n_prefix, int32_t block_len,
                                int32_t block_start, const int32_t* suffix_pos, int32_t n_suffix,
                                const void* embed, int64_t vocab, int32_t hidden, int32_t mask_id,
                                const int32_t* prev_topk_ids, const float* prev_topk_prob,
                                int32_t k, float alpha, void* x_out, int32_t* pos_out,
                                ssm_stream_t stream) {
  ssm_status s = ssm::check_common(embed, vocab, hidden, mask_id, k, alpha, block_len, x_out);
  if (s != SSM_OK) return s;
  if (batch < 0 || n_prefix < 0 || n_suffix < 0 || block_start < 0) return SSM_ERR_INVALID_ARG;
  if (block_len > 0 && !block_tokens) return SSM_ERR_INVALID_ARG;
  if (n_prefix > 0 && !prefix_tokens) return SSM_ERR_INVALID_ARG;
  if (n_suffix > 0 && !suffix_pos) return SSM_ERR_INVALID_ARG;
  if (prev_topk_ids && k > 0 && !prev_topk_prob) return SSM_ERR_INVALID_ARG;
  const int32_t rows = n_prefix + block_len + n_suffix;
  if (batch == 0 || rows == 0) return SSM_OK;
  if (batch > 65535) return SSM_ERR_UNSUPPORTED;
  ssm::BuildParams p{};
  p.problems = nullptr;
  p.n_problems = batch;
  p.u_n_prefix = n_prefix;
  p.u_n_suffix = n_suffix;
  p.u_block_start = block_start;
  p.block_len = block_len;
  p.block_tokens = block_tokens;
  p.prefix_tokens = prefix_tokens;
  p.suffix_pos = suffix_pos;
  p.embed = static_cast<const uint4*>(embed);
  p.vocab = vocab;
  p.hvec = hidden / 8;
  p.mask_id = mask_id;
  p.topk_ids = (k > 0) ? prev_topk_ids : nullptr;
  p.topk_prob = prev_topk_prob;
  p.k = k;
  p.alpha = alpha;
  p.x_out = static_cast<uint4*>(x_out);
  p.pos_out = pos_out;
  p.err = ssm::device_error_word();
  dim3 grid(rows, batch);
  if (ssm::two_columns(static_cast<int64_t>(rows) * batch))
    ssm::launch_k(ssm::build_step_input_kernel<2>, dim3(grid), dim3(ssm::kBuildThreads), 0,
                  reinterpret_cast<cudaStream_t>(stream), p);
  else
    ssm::launch_k(ssm::build_step_input_kernel<1>, dim3(grid), dim3(ssm::kBuildThreads), 0,
                  reinterpret_cast<cudaStream_t>(stream), p);
  return ssm::launch_status();
}

ssm_status ssm_build_step_input_varlen(const ssm_step_problem* problems, int32_t n_problems,
                                       int32_t max_rows, int32_t block_len,
                                       const int32_t* block_tokens, const int32_t* prefix_tokens,
                                       const int32_t* suffix_pos, const void* embed,
                                       int64_t vocab, int32_t hidden, int32_t mask_id,
                                       const int32_t* prev_topk_ids, const float* prev_topk_prob,
                                       int32_t k, float alpha, void* x_out, int32_t* pos_out,
                                       ssm_stream_t stream) {
  ssm_status s = ssm::check_common(embed, vocab, hidden, mask_id, k, alpha, block_len, x_out);
  if (s != SSM_OK) return s;
  if (n_problems < 0 || max_rows < 0) return SSM_ERR_INVALID_ARG;
  if (n_problems == 0 || max_rows == 0) return SSM_OK;
  if (!problems || !suffix_pos || (block_len > 0 && !block_tokens)) return SSM_ERR_INVALID_ARG;
  if (prev_topk_ids && k > 0 && !prev_topk_prob) return SSM_ERR_INVALID_ARG;
  if (n_problems > 65535) return SSM_ERR_UNSUPPORTED;
  ssm::BuildParams p{};
  p.problems = problems;
  p.n_problems = n_problems;
  p.block_len = block_len;
  p.block_tokens = block_tokens;
  p.prefix_tokens = prefix_tokens;
  p.suffix_pos = suffix_pos;
  p.embed = static_cast<const uint4*>(embed);
  p.vocab = vocab;
  p.hvec = hidden / 8;
  p.mask_id = mask_id;
  p.topk_ids = (k > 0) ? prev_topk_ids : nullptr;
  p.topk_prob = prev_topk_prob;
  p.k = k;
  p.alpha = alpha;
  p.x_out = static_cast<uint4*>(x_out);
  p.pos_out = pos_out;
  p.err = ssm::device_error_word();
  dim3 grid(max_rows, n_problems);
  if (ssm::two_columns(static_cast<int64_t>(max_rows) * n_problems))
    ssm::launch_k(ssm::build_step_input_kernel<2>, dim3(grid), dim3(ssm::kBuildThreads), 0,
                  reinterpret_cast<cudaStream_t>(stream), p);
  else
    ssm::launch_k(ssm::build_step_input_kernel<1>, dim3(grid), dim3(ssm::kBuildThreads), 0,
                  reinterpret_cast<cudaStream_t>(stream), p);
  return ssm::launch_status();
}

ssm_status ssm_select_build_step_input_varlen(const ssm_step_problem* problems, const ssm_suffix_cfg* cfgs,
                                              int32_t n_problems, int32_t max_rows, int32_t block_len,
                                              const int32_t* block_tokens, const int32_t* prefix_tokens,
                                              int32_t* suffix_pos_out, const void* embed, int64_t vocab,
                                              int32_t hidden, int32_t mask_id, const int32_t* prev_topk_ids,
                                              const float* prev_topk_prob, int32_t k, float alpha, void* x_out,
                                              int32_t* pos_out, ssm_stream_t stream) {
  ssm_status s = ssm::check_common(embed, vocab, hidden, mask_id, k, alpha, block_len, x_out);
  if (s != SSM_OK) return s;
  if (n_problems < 0 || max_rows < 0) return SSM_ERR_INVALID_ARG;
  if (n_problems == 0 || max_rows == 0) return SSM_OK;
  if (!problems || !cfgs || (block_len > 0 && !block_tokens)) return SSM_ERR_INVALID_ARG;
  if (prev_topk_ids && k > 0 && !prev_topk_prob) return SSM_ERR_INVALID_ARG;
  if (n_problems > 65535) return SSM_ERR_UNSUPPORTED;
  ssm::BuildParams p{};
  p.problems = problems;
  p.n_problems = n_problems;
  p.block_len = block_len;
  p.block_tokens = block_tokens;
  p.prefix_tokens = prefix_tokens;
  p.cfgs = cfgs;
  p.suffix_pos_out = suffix_pos_out;
  p.embed = static_cast<const uint4*>(embed);
  p.vocab = vocab;
  p.hvec = hidden / 8;
  p.mask_id = mask_id;
  p.topk_ids = (k > 0) ? prev_topk_ids : nullptr;
  p.topk_prob = prev_topk_prob;
  p.k = k;
  p.alpha = alpha;
  p.x_out = static_cast<uint4*>(x_out);
  p.pos_out = pos_out;
  p.err = ssm::device_error_word();
  if (ssm::two_columns(static_cast<int64_t>(max_rows) * n_problems))
    ssm::launch_k(ssm::build_step_input_kernel<2>, dim3(max_rows, n_problems), dim3(ssm::kBuildThreads), 0,
                  reinterpret_cast<cudaStream_t>(stream), p);
  else
    ssm::launch_k(ssm::build_step_input_kernel<1>, dim3(max_rows, n_problems), dim3(ssm::kBuildThreads), 0,
                  reinterpret_cast<cudaStream_t>(stream), p);
  return ssm::launch_status();
}

}  // extern "C"
