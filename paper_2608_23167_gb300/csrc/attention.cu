// attention.cu -- bidirectional MHA/GQA attention over prefix cache + current
// block + retained suffix (Sec. 1 and Sec. 2: DLM attention is non-causal;
// Sec. 3.2 "Sparse Input Construction": retained suffix tokens keep their
// original rotary encodings; Table 4 "PC.": prefix K/V come from a cache).
//
// Two kernels:
//  * rope_pack_kernel rotates the new queries and keys at their original
//    positions and packs the queries of one GQA group into one row block,
//    (query i, head-in-group hl) -> row i * grp + hl, so that a 128-row M tile
//    of the tensor-core GEMM holds every query head that shares a K/V head.
//  * attn_fwd_kernel: persistent, one CTA per SM.  Work units are (problem,
//    kv head, pair of 128-row query tiles), (problem, kv head, one tile) or
//    (problem, two kv heads, one tile each), whichever the host's makespan
//    estimate prefers, or, for ragged batches whose problems share one cache
//    prefix, pairs of tiles of consecutive problems' packed rows (each row
//    masked to its own prefix and new rows); they are dealt in snake order, and barrier phases carry over from unit to unit,
//    so the next unit's Q/K loads and first QK^T overlap the current unit's
//    last softmax and epilogue.  Per unit,
//    warps 0 and 2 stream the K and the V tiles with TMA, each ring at its own
//    pace (128 keys = four 32-row sub-boxes, so the cache segment and the
//    new-row segment pack back to back with at most 31 padded keys each;
//    2-stage K ring, 3-stage V ring).  Warp 1 issues tcgen05.mma: S = Q K^T
//    from shared memory into tensor memory, and O += P V with P read from
//    tensor memory; warp 3 waits for the K and V tiles on its behalf.  Two
//    softmax warpgroups ("slots" A and B, one query row per thread) alternate:
//    while one turns its S tile into P (written back over S as bf16), the
//    tensor core runs the other slot's GEMMs.  With two query tiles each slot
//    owns one; with a single query tile the slots split the key tiles
//    (even/odd) and merge their partial softmax states at the end; with two
//    kv heads each slot owns one head's tile and key tiles.  After a
//    slot's first tile of a unit the exponentials are taken against the
//    current reference without a row maximum; O is rescaled only when a
//    tile's row sum of p exceeds 2^16.
#include <cuda_bf16.h>
#include <cudaTypedefs.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "attn_common.cuh"
#include "rope.cuh"
#include "tmem_io.cuh"

namespace ssm {
namespace {

constexpr int kKStages = 2;
constexpr int kVStages = 3;
constexpr uint32_t kOCol = 256;       // O of slot X at 256 + X * D; S (and P) of slot X at X * 128

enum Bar {
  Q_FULL = 0,
  Q_EMPTY = 1,
  K_FULL = 2,
  K_EMPTY = K_FULL + kKStages,
  V_FULL = K_EMPTY + kKStages,
  V_EMPTY = V_FULL + kVStages,
  S_FULL = V_EMPTY + kVStages,  // [2]: one per slot
  P_FULL = S_FULL + 2,          // [2]
  O_DONE = P_FULL + 2,          // [2]
  O_FREE = O_DONE + 2,          // [2]: the epilogue has read the slot's O
  MERGE_FULL = O_FREE + 2,      // split keys: slot B's (max, sum) are in shared memory
  DRAIN = MERGE_FULL + 1,
  N_BARS = DRAIN + 1
};

template <int D>
struct Layout {
  static constexpr int NP = D / 64;                   // 64-column panels per row
  static constexpr int TILE = NP * kPanel;            // one 128-row tile
  static constexpr int Q = 0;                         // two query tiles
  static constexpr int K = Q + 2 * TILE;
  static constexpr int V = K + kKStages * TILE;
  static constexpr int BAR = V + kVStages * TILE;
  static constexpr int MERGE = BAR + N_BARS * 8 + 8;  // split-key merge: (m, l) per row
  static constexpr int BYTES = MERGE + 2 * kBM * 4;
  static constexpr int ALLOC = BYTES + 1024;          // slack to align the base to 1024 B
  static_assert(ALLOC <= 232448, "shared memory budget");
};

// ---------------------------------------------------------------------------
// RoPE + GQA packing of the new rows
// ---------------------------------------------------------------------------

constexpr int kRopeWarps = 8;
constexpr int kRopePasses = 4;  // head passes of a warp in flight (a lane's loads: 2 x this, 16 bytes each)

// Problem whose new rows contain row r: the last problem starting at or before r
// (problems of a packable plan start at increasing rows).
__device__ __forceinline__ int problem_of_row(const ssm_attn_problem* pr, int n_prob, int64_t r) {
  int lo = 0, hi = n_prob - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (pr[mid].new_row <= r) lo = mid; else hi = mid - 1;
  }
  return lo;
}

// The unit plan of a ragged batch (one warp).  Packed units are used when every problem
// reads the same cache rows (the same cache_row), the problems' new rows follow one
// another from row 0 without gaps, and packing needs fewer 128-row query tiles than one
// problem per unit does.
__device__ void attn_plan_warp(const AttnParams& p, int n_prob, int64_t total_new, int max_pairs) {
  const int lane = threadIdx.x & 31;
  const ssm_attn_problem* pr = p.problems;
  const int64_t c0 = pr[0].cache_row;
  bool ok = true;
  int64_t tiles = 0;
  for (int b = lane; b < n_prob; b += 32) {
    const ssm_attn_problem q = pr[b];
    const int64_t expect = b == 0 ? 0 : pr[b - 1].new_row + pr[b - 1].n_new;
    ok = ok && q.cache_row == c0 && q.new_row == expect && q.n_new > 0;
    tiles += (static_cast<int64_t>(q.n_new) * p.grp + kBM - 1) / kBM;
  }
  ok = __all_sync(0xffffffffu, ok);
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) tiles += __shfl_xor_sync(0xffffffffu, tiles, o);
  const int64_t last_end = pr[n_prob - 1].new_row + pr[n_prob - 1].n_new;
  const int64_t qrows = total_new * p.grp;
  const int64_t packed_tiles = (qrows + kBM - 1) / kBM;
  const int n_pairs = static_cast<int>((qrows + 2 * kBM - 1) / (2 * kBM));
  const bool packed = ok && last_end == total_new && packed_tiles < tiles && n_pairs <= max_pairs;
  AttnPlanUnit* units = reinterpret_cast<AttnPlanUnit*>(p.plan + 1);
  if (packed) {
    for (int i = lane; i < n_pairs; i += 32) {
      AttnPlanUnit u;
      const int64_t p0 = static_cast<int64_t>(i) * 2 * kBM;
      u.p0 = static_cast<int32_t>(p0);
      u.rows = static_cast<int32_t>(qrows - p0 < 2 * kBM ? qrows - p0 : 2 * kBM);
      const int b_lo = problem_of_row(pr, n_prob, p0 / p.grp);
      const int b_hi = problem_of_row(pr, n_prob, (p0 + u.rows - 1) / p.grp);
      int c_max = 0;
      for (int b = b_lo; b <= b_hi; ++b) c_max = max(c_max, pr[b].n_cache);
      u.c_max = c_max;
      u.pad = 0;
      u.nr_lo = pr[b_lo].new_row;
      u.nr_hi = pr[b_hi].new_row + pr[b_hi].n_new;
      units[i] = u;
    }
  }
  if (lane == 0) {
    AttnPlanHdr h{};
    h.packed = packed ? 1 : 0;
    h.n_pairs = packed ? n_pairs : 0;
    h.cache_row = c0;
    *p.plan = h;
  }
}

// L2 eviction-priority hints of the pre-pass: the raw rows it reads once go first, the rotated
// rows it writes (which the forward reads next) stay longest, so that more of them are still in L2,
// not yet written back, when the forward starts; their write-back then falls into the forward's
// time, whose DRAM traffic is a fifth of the copy bandwidth.
__device__ __forceinline__ uint64_t l2_policy_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_policy_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint4 ld_l2_hint(const void* ptr, uint64_t pol) {
  uint4 v;
  asm volatile("ld.global.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(ptr), "l"(pol));
  return v;
}
__device__ __forceinline__ void st_l2_hint(void* ptr, const uint4& v, uint64_t pol) {
  asm volatile("st.global.L2::cache_hint.v4.u32 [%0], {%1, %2, %3, %4}, %5;" ::"l"(ptr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w), "l"(pol)
               : "memory");
}

// Persistent warps over (problem, row, head part) items, item = (problem *
// rows_per_problem_max + row) * hsplit + part (items past a problem's row count are
// skipped).  A row's head vectors are cut into hsplit parts of hper vectors (whole head
// passes): one part per row on large batches, several on small ones, so that the rows of a
// small batch still spread over every warp instead of each warp walking all of its row's
// passes one memory round trip after another.  A row's D/2 angles are formed per item (two
// per lane) and shared through shared memory; a lane then owns eight rotation pairs
// (i, i + D/2) of one head vector (D/16 lanes per head, 16-byte loads and stores,
// kRopePasses head passes in flight; the first pass's loads are issued before the angles are
// formed).  The rotation is rope.cuh's (inverse frequencies from the host).
template <int D>
__global__ void __launch_bounds__(kRopeWarps * 32, 3) rope_pack_kernel(
    const __nv_bfloat16* __restrict__ q, const __nv_bfloat16* __restrict__ k,
    const int32_t* __restrict__ pos, AttnParams p, const RopeFreqs<D> freqs, int32_t rows_per_problem_max,
    int32_t n_prob,
    int32_t max_pairs, int32_t hsplit, int32_t hper, __nv_bfloat16* __restrict__ qhat,
    __nv_bfloat16* __restrict__ khat) {
  pdl_enter();
  constexpr int LPH = D / 16;       // lanes per head vector: eight rotation pairs per lane
  constexpr int HPP = 32 / LPH;     // head vectors per warp pass
  __shared__ uint64_t turn[D / 2];
  __shared__ float s_cs[kRopeWarps][D / 2], s_sn[kRopeWarps][D / 2];
  if (threadIdx.x < D / 2) turn[threadIdx.x] = freqs.turn[threadIdx.x];
  __syncthreads();
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (p.plan && blockIdx.x == 0 && warp == 0) attn_plan_warp(p, n_prob, p.new_rows_extent, max_pairs);
  const int sub = lane % LPH, hoff = lane / LPH;
  const int n_vec = p.h_q + p.h_kv;
  const int64_t total = static_cast<int64_t>(n_prob) * rows_per_problem_max * hsplit;
  const uint64_t pol_in = l2_policy_evict_first(), pol_out = l2_policy_evict_last();
  for (int64_t it = static_cast<int64_t>(blockIdx.x) * kRopeWarps + warp; it < total;
       it += static_cast<int64_t>(gridDim.x) * kRopeWarps) {
    const int64_t rit = it / hsplit;
    const int part = static_cast<int>(it - rit * hsplit);
    const int prob = static_cast<int>(rit / rows_per_problem_max);
    const int i = static_cast<int>(rit - static_cast<int64_t>(prob) * rows_per_problem_max);
    const Geom gm = problem_geom(p, prob);
    if (i >= gm.n_new) continue;
    const int64_t row = gm.new_row + i;
    const int hbeg = part * hper, hend = min(n_vec, hbeg + hper);
    const int32_t ps = pos[p.problems ? row : i];
    uint4 x1[kRopePasses], x2[kRopePasses];
    auto load_pass = [&](int h0) {
#pragma unroll
      for (int u = 0; u < kRopePasses; ++u) {
        const int h = h0 + u * HPP;
        if (h < hend) {
          const __nv_bfloat16* src = h < p.h_q ? q + (row * p.h_q + h) * D : k + (row * p.h_kv + (h - p.h_q)) * D;
          x1[u] = ld_l2_hint(src + 8 * sub, pol_in);
          x2[u] = ld_l2_hint(src + D / 2 + 8 * sub, pol_in);
        }
      }
    };
    load_pass(hbeg + hoff);
    // each pair's angle once per item (a lane takes pairs lane, lane + 32), shared through shared memory
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
    // a packed unit's softmax rows read their problem's key bounds from here in one load: the
    // cache prefix length and the problem's new rows [new_row, new_row + n_new)
    if (p.row_bounds && part == 0 && lane == 0)
      p.row_bounds[row] = make_int4(gm.n_cache, static_cast<int>(gm.new_row), static_cast<int>(gm.new_row + gm.n_new), 0);
    for (int h0 = hbeg + hoff; h0 < hend; h0 += kRopePasses * HPP) {
      if (h0 != hbeg + hoff) load_pass(h0);
#pragma unroll
      for (int u = 0; u < kRopePasses; ++u) {
        const int h = h0 + u * HPP;
        if (h >= hend) continue;
        uint2 ya, yb, yc, yd;
        rope_rotate4(make_uint2(x1[u].x, x1[u].y), make_uint2(x2[u].x, x2[u].y), cs0, sn0, ya, yb);
        rope_rotate4(make_uint2(x1[u].z, x1[u].w), make_uint2(x2[u].z, x2[u].w), cs1, sn1, yc, yd);
        __nv_bfloat16* dst;
        if (h < p.h_q) {
          // queries packed by GQA group: a uniform batch per (problem, kv head); a ragged batch
          // head-major over all new rows (the query tiles of consecutive problems then adjoin)
          const int g = h / p.grp, hl = h - g * p.grp;
          const int64_t dst_row =
              p.problems ? static_cast<int64_t>(g) * p.qrows_g + row * p.grp + hl
                         : (gm.new_row * p.h_kv + static_cast<int64_t>(g) * gm.n_new) * p.grp +
                               static_cast<int64_t>(i) * p.grp + hl;
          dst = qhat + dst_row * D;
        } else {
          dst = khat + (row * p.h_kv + (h - p.h_q)) * D;
        }
        st_l2_hint(dst + 8 * sub, make_uint4(ya.x, ya.y, yc.x, yc.y), pol_out);
        st_l2_hint(dst + D / 2 + 8 * sub, make_uint4(yb.x, yb.y, yd.x, yd.y), pol_out);
      }
    }
  }
}

// ---------------------------------------------------------------------------
// Attention forward
// ---------------------------------------------------------------------------

// One work unit: a pair of query tiles of one kv head, either of one problem or, with
// packed units, of the packed rows of consecutive problems (gm then describes the
// unit's key stream: the shared cache prefix [0, c_max) and the new rows [nr_lo, nr_hi)).
struct Unit {
  Geom gm;
  int prob, g, qt0, n_csub, n_nsub, nt;
  int urows;      // query rows (query x head-in-group) of the unit from its first tile on
  int64_t orow0;  // packed row of the unit's first query: query = packed / grp, head-in-group = packed % grp
  int64_t qrow0;  // ragged batches: its row in the kv head's block of the rotated queries
  bool two, valid, packed;
  bool dual;      // two kv heads (g, g + 1) of one problem, one query tile each: slot X takes head g + X
};

// Ring entries (K or V tiles) a unit streams: its key tiles, twice over for a dual-head unit
// (entry e is key tile e / 2 of head g + e % 2, so the slots' tiles alternate in the rings).
__device__ __forceinline__ int unit_entries(const struct Unit& w) { return w.dual ? 2 * w.nt : w.nt; }

// Units are dealt to the persistent CTAs in waves of gridDim.x, each wave in the opposite
// direction to the last ("snake" order): with units sorted by decreasing cost, a CTA that took
// a heavy unit in one wave takes a light one in the next, which evens out the CTAs' totals
// (on the long sweep the simulated makespan falls from 9 % to 6 % above the mean).  Every
// role of a CTA walks the same sequence; it is increasing, so the first unit past the end
// ends the walk.
__device__ __forceinline__ int snake_unit(int k) {
  const int c = static_cast<int>(blockIdx.x), g = static_cast<int>(gridDim.x);
  return k * g + ((k & 1) ? g - 1 - c : c);
}

// The kernel-wide unit plan: packed units from the device plan, else problem units.
struct UnitPlan {
  bool packed;
  int n_pairs, total_units;
  int64_t cache_row;
};

// PACKABLE = false compiles the kernel without packed units at all (no plan read, no per-row
// key bounds in the softmax): the host launches that form for batches that cannot pack.
template <bool PACKABLE>
__device__ __forceinline__ UnitPlan read_plan(const AttnParams& p) {
  UnitPlan up{false, 0, p.total_units, 0};
  if (PACKABLE && p.plan) {
    const AttnPlanHdr h = *p.plan;
    if (h.packed) {
      up.packed = true;
      up.n_pairs = h.n_pairs;
      up.total_units = h.n_pairs * p.h_kv;
      up.cache_row = h.cache_row;
    }
  }
  return up;
}

// DUAL = false compiles out the dual-head units (the packable form of the kernel never takes them).
template <bool DUAL>
__device__ __forceinline__ Unit make_unit(const AttnParams& p, const UnitPlan& up, int u) {
  Unit w;
  if (up.packed) {
    // most keys first: pairs in decreasing order (a later pair's problems have longer prefixes
    // in a block sweep), the kv heads of one pair on neighbouring CTAs (shared K/V in L2)
    const int pair_rev = u / p.h_kv;
    w.g = u - pair_rev * p.h_kv;
    const AttnPlanUnit pu = reinterpret_cast<const AttnPlanUnit*>(p.plan + 1)[up.n_pairs - 1 - pair_rev];
    w.prob = -1;
    w.gm.new_row = pu.nr_lo;
    w.gm.cache_row = up.cache_row;
    w.gm.n_new = static_cast<int32_t>(pu.nr_hi - pu.nr_lo);
    w.gm.n_cache = pu.c_max;
    w.qt0 = 0;
    w.urows = pu.rows;
    w.orow0 = pu.p0;
    w.qrow0 = pu.p0;
    w.valid = true;
    w.two = pu.rows > kBM;
    w.packed = true;
    w.dual = false;
  } else if (DUAL && p.dual_heads) {
    // two kv heads of one problem, one query tile each (the host takes this form only when every
    // problem's query rows fit one tile and h_kv is even)
    const int hp = p.h_kv / 2;
    w.prob = u / hp;
    w.g = 2 * (u - w.prob * hp);
    w.gm = problem_geom(p, w.prob);
    w.qt0 = 0;
    w.urows = w.gm.n_new * p.grp;
    w.orow0 = w.gm.new_row * p.grp;
    w.qrow0 = w.orow0;
    w.valid = w.urows > 0;
    w.two = false;
    w.packed = false;
    w.dual = true;
  } else {
    const int pg = u / p.units_per_pg;
    const int pair = u - pg * p.units_per_pg;
    w.prob = pg / p.h_kv;
    w.g = pg - w.prob * p.h_kv;
    w.gm = problem_geom(p, w.prob);
    const int rows_q = w.gm.n_new * p.grp;
    const int n_qt = (rows_q + kBM - 1) / kBM;
    w.qt0 = p.tiles_per_unit * pair;
    w.urows = rows_q - w.qt0 * kBM;
    w.orow0 = w.gm.new_row * p.grp + w.qt0 * kBM;
    w.qrow0 = w.orow0;
    w.valid = w.qt0 < n_qt;
    w.two = p.tiles_per_unit == 2 && w.qt0 + 1 < n_qt;
    w.packed = false;
    w.dual = false;
  }
  w.n_csub = (w.gm.n_cache + kSub - 1) / kSub;
  w.n_nsub = (w.gm.n_new + kSub - 1) / kSub;
  w.nt = (w.n_csub + w.n_nsub + 3) / 4;
  return w;
}

// DUAL compiles the dual-head units in (only without packed units): a separate form, so that the
// other forms carry none of their code.
template <int D, bool PACKABLE, bool POLL, bool DUAL>
__global__ void __launch_bounds__(kAttnThreads, 1) attn_fwd_kernel(
    const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_kc,
    const __grid_constant__ CUtensorMap tm_vc, const __grid_constant__ CUtensorMap tm_kn,
    const __grid_constant__ CUtensorMap tm_vn, const __grid_constant__ CUtensorMap tm_kc128,
    const __grid_constant__ CUtensorMap tm_vc128, const __grid_constant__ CUtensorMap tm_kn128,
    const __grid_constant__ CUtensorMap tm_vn128, const AttnParams p) {
  pdl_enter();
  using L = Layout<D>;
  constexpr int NP = L::NP;
  constexpr uint32_t kIdescQK = idesc_bf16_f32(kBM, kBN, false, false);
  constexpr uint32_t kIdescPV = idesc_bf16_f32(kBM, D, false, true);

  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + N_BARS);
  float* merge_buf = reinterpret_cast<float*>(smem + L::MERGE);  // [m | l][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool uniform = p.problems == nullptr;
  const UnitPlan up = read_plan<PACKABLE>(p);

  // No control flow in this kernel depends on the lane: each warp walks its loop
  // as one converged path and a single lane issues through predicated
  // instructions (the *_if helpers), so every warp reaches the .sync.aligned
  // TMEM instructions, tcgen05.dealloc and the CTA barriers whole.
  const bool leader = lane == 0;
  if (warp == 0) {
    mbar_init_if(leader, &bars[Q_FULL], 1);
    mbar_init_if(leader, &bars[Q_EMPTY], 1);
    for (int s = 0; s < kKStages; ++s) {
      mbar_init_if(leader, &bars[K_FULL + s], 1);
      mbar_init_if(leader, &bars[K_EMPTY + s], 1);
    }
    for (int s = 0; s < kVStages; ++s) {
      mbar_init_if(leader, &bars[V_FULL + s], 1);
      mbar_init_if(leader, &bars[V_EMPTY + s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init_if(leader, &bars[S_FULL + x], 1);
      mbar_init_if(leader, &bars[P_FULL + x], 5);   // one arrival per softmax warp, one from the K/V watcher
      mbar_init_if(leader, &bars[O_DONE + x], 1);
      mbar_init_if(leader, &bars[O_FREE + x], 4);
    }
    mbar_init_if(leader, &bars[MERGE_FULL], 4);
    mbar_init_if(leader, &bars[DRAIN], 1);
    fence_mbar_init();
    tma_prefetch_desc(&tm_q);
    tma_prefetch_desc(&tm_kc);
    tma_prefetch_desc(&tm_vc);
    tma_prefetch_desc(&tm_kn);
    tma_prefetch_desc(&tm_vn);
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish_alloc_permit();
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp < 4) {
    // warpgroup 0 gives registers back (all four warps, one instruction)
    setmaxnreg_dec<kCtrlRegs>();
    if (warp == 0 || warp == 2) {
      // ------------------------------------------------------------- TMA producers
      // warp 0 loads Q and the K ring, warp 2 the V ring, each at its own pace
      const int half = warp == 2 ? 1 : 0;
      bool ok = true;
      int qcount = 0;  // units whose Q was loaded
      int fills = 0;   // tiles loaded into this ring so far (all units)
      const int nst = half ? kVStages : kKStages;
      for (int k_u = 0, u = snake_unit(0); u < up.total_units && ok; u = snake_unit(++k_u)) {
        const Unit w = make_unit<DUAL>(p, up, u);
        if (!w.valid) continue;
        if (!half) {
          if (qcount > 0) ok = warp_wait<POLL>(&bars[Q_EMPTY], (qcount - 1) & 1, p.wait_ns);
          if (!ok) break;
          const int nq = (w.two || w.dual) ? 2 : 1;
          mbar_arrive_expect_tx_if(leader, &bars[Q_FULL], nq * L::TILE);
          for (int x = 0; x < nq; ++x) {
            // a pair: tiles qt0 and qt0 + 1 of kv head g; dual heads: tile qt0 of heads g and g + 1
            const int gx = w.g + (w.dual ? x : 0);
            const int tx = w.dual ? 0 : x;
            int qy, qz;
            if (uniform) {
              qy = (w.qt0 + tx) * kBM;
              qz = w.prob * p.h_kv + gx;
            } else {
              qy = static_cast<int>(static_cast<int64_t>(gx) * p.qrows_g + w.qrow0) + tx * kBM;
              qz = 0;
            }
#pragma unroll
            for (int pn = 0; pn < NP; ++pn)
              tma_load_3d_if(leader, smem + L::Q + x * L::TILE + pn * kPanel, &tm_q, &bars[Q_FULL], pn * 64, qy,
                             qz);
          }
          ++qcount;
        }
        const int c3 = uniform ? w.prob : 0;
        const int ne = unit_entries(w);
        for (int e = 0; e < ne && ok; ++e) {
          const int jt = w.dual ? (e >> 1) : e;            // key tile
          const int gh = w.g + (w.dual ? (e & 1) : 0);     // its kv head
          const int st = fills % nst, fill = fills / nst;
          if (fill > 0) ok = warp_wait<POLL>(&bars[(half ? V_EMPTY : K_EMPTY) + st], (fill - 1) & 1, p.wait_ns);
          if (!ok) break;
          uint64_t* full = &bars[(half ? V_FULL : K_FULL) + st];
          mbar_arrive_expect_tx_if(leader, full, L::TILE);
          uint8_t* dst = smem + (half ? L::V : L::K) + st * L::TILE;
          const int sub0 = 4 * jt;
          const bool whole_cache = sub0 + 3 < w.n_csub && (sub0 + 4) * kSub <= w.gm.n_cache;
          const bool whole_new = sub0 >= w.n_csub && (sub0 - w.n_csub + 4) * kSub <= w.gm.n_new;
          if (whole_cache || whole_new) {
            const CUtensorMap* map = whole_cache ? (half ? &tm_vc128 : &tm_kc128) : (half ? &tm_vn128 : &tm_kn128);
            const int c2 = whole_cache ? (uniform ? sub0 * kSub : static_cast<int>(w.gm.cache_row + sub0 * kSub))
                                       : (uniform ? (sub0 - w.n_csub) * kSub
                                                  : static_cast<int>(w.gm.new_row + (sub0 - w.n_csub) * kSub));
#pragma unroll
            for (int pn = 0; pn < NP; ++pn) tma_load_4d_if(leader, dst + pn * kPanel, map, full, pn * 64, gh, c2, c3);
          } else {
#pragma unroll
            for (int sb = 0; sb < 4; ++sb) {
              const int sub = 4 * jt + sb;
              const CUtensorMap* map;
              int c2;
              if (sub < w.n_csub) {
                map = half ? &tm_vc : &tm_kc;
                c2 = uniform ? sub * kSub : static_cast<int>(w.gm.cache_row + sub * kSub);
              } else if (sub - w.n_csub < w.n_nsub) {
                map = half ? &tm_vn : &tm_kn;
                c2 = uniform ? (sub - w.n_csub) * kSub : static_cast<int>(w.gm.new_row + (sub - w.n_csub) * kSub);
              } else {
                map = half ? &tm_vn : &tm_kn;  // beyond both segments: an out-of-range box reads zeros
                c2 = p.new_rows_extent;
              }
#pragma unroll
              for (int pn = 0; pn < NP; ++pn)
                tma_load_4d_if(leader, dst + pn * kPanel + sb * kSub * 128, map, full, pn * 64, gh, c2, c3);
            }
          }
          ++fills;
        }
      }
      if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
      // Every copy in flight lands before the CTA's shared memory is released, on every
      // path: the newest fill of each stage is the only one that can still be in flight
      // (an older fill's stage was refilled only after its EMPTY phase, i.e. after it had
      // landed and been consumed).  A consumer that timed out may have left this warp's last
      // fills unconsumed even when this warp itself finished; in a run without timeouts they
      // have all landed and each test below passes at once.  The bound is fixed (kDrainNs),
      // not the wait limit, which a caller may have shortened.
      if (!half && qcount > 0) warp_wait<POLL>(&bars[Q_FULL], (qcount - 1) & 1, kDrainNs);
      for (int i = max(0, fills - nst); i < fills; ++i)
        warp_wait<POLL>(&bars[(half ? V_FULL : K_FULL) + i % nst], (i / nst) & 1, kDrainNs);
    } else if (warp == 1) {
      // ------------------------------------------------------------- MMA issuer
      bool ok = true;
      // operand descriptors: the per-instruction ones differ only in the start address field
      const uint64_t dQ = sdesc_sw128(smem_u32(smem + L::Q), 16, 1024);
      const uint64_t dK = sdesc_sw128(smem_u32(smem + L::K), 16, 1024);
      const uint64_t dV = sdesc_sw128(smem_u32(smem + L::V), kPanel, 1024);
      int ucount = 0;            // units processed
      int kbase = 0, vbase = 0;  // global index of the unit's first K / V tile
      int pv0 = 0, pv1 = 0;      // PV GEMMs issued per slot (all units)
      for (int k_u = 0, u = snake_unit(0); u < up.total_units && ok; u = snake_unit(++k_u)) {
        const Unit w = make_unit<DUAL>(p, up, u);
        if (!w.valid) continue;
        ok = warp_wait<POLL>(&bars[Q_FULL], ucount & 1, p.wait_ns);
        if (!ok) break;
        int kx0 = 0, kx1 = 0;        // jobs issued per slot in this unit
        int jlast0 = 0, jlast1 = 0;  // key tile of each slot's latest QK^T
        bool freed0 = false, freed1 = false;
        // one O_FREE wait per slot and unit: the previous unit's epilogue has read this slot's O
        auto wait_o_free = [&](int x) -> bool {
          bool& f = x ? freed1 : freed0;
          if (f) return true;
          f = true;
          return ucount == 0 || warp_wait<POLL>(&bars[O_FREE + x], (ucount - 1) & 1, p.wait_ns);
        };
        // O_X += P_X V(j) for slot X's latest job
        auto issue_pv = [&](int x) -> bool {
          const int jp = x ? jlast1 : jlast0, k = (x ? kx1 : kx0) - 1;
          int& pv = x ? pv1 : pv0;
          if (!wait_o_free(x)) return false;
          // the K/V watcher's share of this phase vouches for V(jp) and this slot's next K tile
          const int vi = vbase + jp;
          const uint64_t vb = dV + static_cast<uint64_t>(((vi % kVStages) * L::TILE) >> 4);
          const uint32_t d_tmem = tmem + kOCol + x * D, a_tmem = tmem + x * kBN;
          const uint32_t acc0 = k > 0 ? 1u : 0u;
          if (!warp_wait<POLL>(&bars[P_FULL + x], pv & 1, p.wait_ns)) return false;
          tc_fence_after_sync();
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk)
            umma_bf16_ts_if(leader, d_tmem, a_tmem + kk * 8, vb + static_cast<uint64_t>((kk * 16 * 128) >> 4),
                            kIdescPV, kk > 0 ? 1u : acc0);
          umma_commit_if(leader, &bars[O_DONE + x]);
          if (!w.two || x == 1) umma_commit_if(leader, &bars[V_EMPTY + vi % kVStages]);
          ++pv;
          return true;
        };
        // jobs alternate between the slots; j is the job's ring entry (a pair shares each entry)
        const int n_jobs = w.two ? 2 * w.nt : unit_entries(w);
        for (int t = 0; t < n_jobs && ok; ++t) {
          const int x = t & 1;
          const int j = w.two ? (t >> 1) : t;
          const int ki = kbase + j;
          const uint64_t qb = dQ + static_cast<uint64_t>((((w.two || w.dual) ? x : 0) * L::TILE) >> 4);
          const uint64_t kb = dK + static_cast<uint64_t>(((ki % kKStages) * L::TILE) >> 4);
          const uint32_t s_tmem = tmem + x * kBN;
          if ((x ? kx1 : kx0) > 0) {
            // the watcher's share of P_FULL vouches for this slot's next K tile too; issue_pv's
            // fence after that wait orders this QK^T as well
            ok = issue_pv(x);
          } else {
            ok = warp_wait<POLL>(&bars[K_FULL + ki % kKStages], (ki / kKStages) & 1, p.wait_ns);
            if (ok) tc_fence_after_sync();
          }
          if (!ok) break;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint64_t off = static_cast<uint64_t>(((kk >> 2) * kPanel + (kk & 3) * 32) >> 4);
            umma_bf16_ss_if(leader, s_tmem, qb + off, kb + off, kIdescQK, kk > 0 ? 1u : 0u);
          }
          umma_commit_if(leader, &bars[S_FULL + x]);
          if (!w.two || x == 1) umma_commit_if(leader, &bars[K_EMPTY + ki % kKStages]);
          if (x) { jlast1 = j; ++kx1; } else { jlast0 = j; ++kx0; }
        }
        if (ok) umma_commit_if(leader, &bars[Q_EMPTY]);
        if (ok && kx0 > 0) ok = issue_pv(0);
        if (ok && kx1 > 0) ok = issue_pv(1);
        if (ok) ok = wait_o_free(0) && wait_o_free(1);
        kbase += unit_entries(w);
        vbase += unit_entries(w);
        ++ucount;
      }
      if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
      // every issued MMA completes before tensor memory is released
      umma_commit_if(leader, &bars[DRAIN]);
      warp_wait<POLL>(&bars[DRAIN], 0, kDrainNs);
    } else {
      // ------------------------------------------------------------- K/V watcher (warp 3)
      // Every mbarrier test costs the MMA-issuing warp ~150 cycles in which it issues
      // nothing, so this warp takes the K and V waits off it: it walks the issuer's step
      // order and, for each PV, waits until that PV's V tile and the K tile of the slot's
      // next QK^T have landed, then adds its arrival to the slot's P_FULL phase (after
      // seeing the slot's previous phase complete, so it never arrives twice in one phase).
      // The issuer waits for K itself only for a slot's first tile of a unit.  A parity
      // wait is exact only while the barrier cannot be two phases from the awaited one:
      // V tiles are confirmed in ring order and each is released only after a PV this
      // warp vouched for; for K, the fill before the awaited one is known from the slot's
      // QK^T completions, which this warp observes in order (comment in vouch).
      bool ok = true;
      int kbase = 0;
      int done0 = 0, done1 = 0;  // P_FULL phases this warp has arrived on, per slot
      int vconf = 0;             // V tiles (all units) confirmed landed, in order
      // one arrival for slot x's PV of tile jp
      auto vouch = [&](int x, int jp, int jk) -> bool {
        int& d = x ? done1 : done0;
        if (d > 0 && !warp_wait<POLL>(&bars[P_FULL + x], (d - 1) & 1, p.wait_ns)) return false;
        // slot x's d-th QK^T (on K tile jp) has completed, so tile jp has landed; every S
        // of each slot is seen here in order, so the fill before any K tile waited for
        // below is known to have landed (split keys: tile jp itself; both slots on every
        // tile: tile jp - 1, or the previous unit's last tile), and the fill after it
        // needs this vouch: each parity wait stays within its two-phase window
        if (!warp_wait<POLL>(&bars[S_FULL + x], d & 1, p.wait_ns)) return false;
        for (; vconf <= kbase + jp; ++vconf)
          if (!warp_wait<POLL>(&bars[V_FULL + vconf % kVStages], (vconf / kVStages) & 1, p.wait_ns)) return false;
        if (jk >= 0) {
          const int ki = kbase + jk;
          if (!warp_wait<POLL>(&bars[K_FULL + ki % kKStages], (ki / kKStages) & 1, p.wait_ns)) return false;
        }
        mbar_arrive_if(leader, &bars[P_FULL + x]);
        ++d;
        return true;
      };
      for (int k_u = 0, u = snake_unit(0); u < up.total_units && ok; u = snake_unit(++k_u)) {
        const Unit w = make_unit<DUAL>(p, up, u);
        if (!w.valid) continue;
        int kx0 = 0, kx1 = 0, jlast0 = 0, jlast1 = 0;
        const int n_jobs = w.two ? 2 * w.nt : unit_entries(w);
        for (int t = 0; t < n_jobs && ok; ++t) {
          const int x = t & 1;
          const int j = w.two ? (t >> 1) : t;
          if ((x ? kx1 : kx0) > 0) ok = vouch(x, x ? jlast1 : jlast0, j);
          if (x) { jlast1 = j; ++kx1; } else { jlast0 = j; ++kx0; }
        }
        if (ok && kx0 > 0) ok = vouch(0, jlast0, -1);
        if (ok && kx1 > 0) ok = vouch(1, jlast1, -1);
        kbase += unit_entries(w);
      }
      if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
    }
  } else {
    // ------------------------------------------------------------- softmax slots (warps 4..11, warpgroups 1 and 2)
    setmaxnreg_inc<kSoftmaxRegs>();
    const int x = (warp - 4) >> 2;   // slot
    const int quarter = warp & 3;    // TMEM lanes 32*quarter .. +31 belong to this warp
    const int row = quarter * 32 + lane;
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t tS = tmem + lane_off + x * kBN;
    const uint32_t tO = tmem + lane_off + kOCol + x * D;
    const uint32_t tOB = tmem + lane_off + kOCol + D;  // slot B's accumulator (split keys)
    bool ok = true;
    int sj = 0;       // S tiles consumed by this slot (all units)
    int merges = 0;   // split-key merges done
    for (int k_u = 0, u = snake_unit(0); u < up.total_units && ok; u = snake_unit(++k_u)) {
      const Unit w = make_unit<DUAL>(p, up, u);
      if (!w.valid) continue;
      const int jobs = (w.two || w.dual) ? w.nt : (x == 0 ? (w.nt + 1) / 2 : w.nt / 2);
      float m_run = -INFINITY, l_run = 0.f;
      // this thread's query row within the unit; with packed units, its own problem's keys:
      // cache rows below lim, new rows [nlo, nhi) (rows past the unit's end see every key;
      // their outputs are not stored).  Loads are clamped in range rather than branched around.
      const int pr_u = (w.two ? x : 0) * kBM + row;
      // (new rows counted from the unit's first new row, which fits 32 bits)
      int lim = w.gm.n_cache, nlo = 0, nhi = w.gm.n_new;
      if (w.packed) {
        const bool mine = pr_u < w.urows;
        const int4 bd = p.row_bounds[(w.orow0 + min(pr_u, w.urows - 1)) / p.grp];
        lim = mine ? bd.x : lim;
        nlo = mine ? bd.y - static_cast<int>(w.gm.new_row) : nlo;
        nhi = mine ? bd.z - static_cast<int>(w.gm.new_row) : nhi;
      }
      for (int k = 0; k < jobs; ++k) {
        const int j = (w.two || w.dual) ? k : 2 * k + x;
        // The tile's masking plan is made while the tensor core still computes S (it depends
        // only on the tile index and the row's bounds): valid keys of each 32-key sub-box of
        // the tile for this row, columns [lo, hi)
        int lo[4], hi[4];
        bool full_row;
        if (w.packed) {
          full_row = row_sub_bounds(j, w.n_csub, w.n_nsub, lim, nlo, nhi, lo, hi);
        } else {
          full_row = tile_valid_counts(j, w.n_csub, w.n_nsub, w.gm, hi);
#pragma unroll
          for (int s4 = 0; s4 < 4; ++s4) lo[s4] = 0;
        }
        const bool full_tile = __all_sync(0xffffffffu, full_row);
        // A row sees all keys of most sub-boxes or none of them (a whole sub-box of another
        // problem's new rows, or of cache rows past its prefix): the exponent's addend carries
        // that (-inf: none), with no per-key work.  Only in a sub-box that some row of the warp
        // sees in part (votes, warp-uniform) are the invalid keys set to -inf one by one; a row
        // maximum (first tile of a unit, exact path) takes every sub-box masked.
        bool whole = true;
#pragma unroll
        for (int s4 = 0; s4 < 4; ++s4) whole = whole && ((lo[s4] == 0 && hi[s4] == kSub) || hi[s4] <= lo[s4]);
        const bool part_keys = !__all_sync(0xffffffffu, whole);
        uint32_t an_bits = 0;
#pragma unroll
        for (int s4 = 0; s4 < 4; ++s4)
          an_bits |= ((lo[s4] == 0 && hi[s4] == kSub) || hi[s4] <= lo[s4] ? 1u : 0u) << s4;
        an_bits = __reduce_and_sync(0xffffffffu, an_bits);
        ok = warp_wait<POLL>(&bars[S_FULL + x], sj & 1, p.wait_ns);
        if (!ok) break;
        tc_fence_after_sync();
        uint32_t sr[kBN];
        auto load_s = [&](bool for_max) {
          tmem_ld_x128(tS, sr);
          if (for_max ? !full_tile : part_keys) {
#pragma unroll
            for (int s4 = 0; s4 < 4; ++s4) {
              if (!for_max && (an_bits & (1u << s4))) continue;
#pragma unroll
              for (int cc = 0; cc < kSub; ++cc)
                sr[s4 * kSub + cc] =
                    (cc >= lo[s4] && cc < hi[s4]) ? sr[s4 * kSub + cc] : __float_as_uint(-INFINITY);
            }
          }
        };
        load_s(k == 0);
        const float sc = p.scale_log2;
        // row maximum of the tile's scores: eight independent chains of 3-input max, then a short tree
        auto row_max = [&]() -> float {
          float mx8[8];
#pragma unroll
          for (int c = 0; c < 8; ++c) mx8[c] = __uint_as_float(sr[c]);
#pragma unroll
          for (int c = 8; c < kBN; c += 2)
            mx8[(c >> 1) & 7] = fmax3(mx8[(c >> 1) & 7], __uint_as_float(sr[c]), __uint_as_float(sr[c + 1]));
          return fmaxf(fmax3(mx8[0], mx8[1], mx8[2]), fmax3(fmax3(mx8[3], mx8[4], mx8[5]), mx8[6], mx8[7]));
        };
        // p = 2^(s * scale * log2 e - m) into pk (bf16 pairs): packed pair FMA, two MUFU ex2, packed
        // pair sums; returns the row's sum of p over the tile
        uint32_t pk[kBN / 2];
        auto exp_pass = [&](float m) -> float {
          float add[4];
#pragma unroll
          for (int s4 = 0; s4 < 4; ++s4) add[s4] = hi[s4] <= lo[s4] ? -INFINITY : -m;
          float ra[4] = {0.f, 0.f, 0.f, 0.f}, rb[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
          for (int c = 0; c < kBN / 2; ++c) {
            float t0, t1;
            const float a0 = add[c / (kSub / 2)];
            ffma2(t0, t1, __uint_as_float(sr[2 * c]), __uint_as_float(sr[2 * c + 1]), sc, sc, a0, a0);
            const float a = ex2_approx(t0), b = ex2_approx(t1);
            fadd2_acc(ra[c & 3], rb[c & 3], a, b);
            pk[c] = pack_bf16x2(a, b);
          }
          return ((ra[0] + rb[0]) + (ra[1] + rb[1])) + ((ra[2] + rb[2]) + (ra[3] + rb[3]));
        };
        float lt;
        if (k == 0) {
          // the slot's first tile of the unit sets the reference m: its row maximum (0 for a row
          // with no valid key in this tile, which packed units can give: its first p are then 0)
          const float mx0 = row_max();
          m_run = mx0 == -INFINITY ? 0.f : mx0 * sc;
          lt = exp_pass(m_run);
        } else {
          // later tiles: exponentials against the current reference without a row maximum.
          // A tile sum of at most 2^16 bounds every p by 2^16 (far inside fp32 / bf16 range);
          // a row above it (or inf / NaN) takes the exact path: new m from the row maximum,
          // O and l rescaled by 2^(m_old - m_new), exponentials again.  Branch-free per row
          // (selects only): the warp stays converged for the TMEM accesses.
          lt = exp_pass(m_run);
          const bool need = !(lt <= kSpecSumMax);
          if (__any_sync(0xffffffffu, need)) {
            // S is still in tensor memory (P has not been written over it): load it again
            // rather than keep the scores live through the exponentials
            load_s(true);
            const float m_new = fmaxf(m_run, row_max() * sc);
            const float alpha = ex2_approx(need ? m_run - m_new : 0.f);
            // the previous PV of this slot completed before this S tile was committed
            ok = warp_wait<POLL>(&bars[O_DONE + x], (sj - 1) & 1, p.wait_ns);
            if (!ok) break;
            tc_fence_after_sync();
#pragma unroll
            for (int ch = 0; ch < D / 32; ++ch) {
              uint32_t o[32];
              tmem_ld_x32(tO + ch * 32, o);
#pragma unroll
              for (int c = 0; c < 32; ++c) o[c] = __float_as_uint(__uint_as_float(o[c]) * alpha);
              tmem_st_x32(tO + ch * 32, o);
            }
            l_run *= alpha;
            m_run = need ? m_new : m_run;
            lt = exp_pass(m_run);
          }
        }
        l_run += lt;
        // P (bf16) overwrites the first 64 columns of this slot's S; the PV GEMM reads it from there
        tmem_st_x64(tS, pk);
        tc_fence_before_sync();
        warp_arrive(&bars[P_FULL + x]);
        ++sj;
      }
      // the slot's last PV of this unit (it completes before any later S of this slot)
      if (ok && jobs > 0) ok = warp_wait<POLL>(&bars[O_DONE + x], (sj - 1) & 1, p.wait_ns);
      if (!ok) break;
      tc_fence_after_sync();
      // Split keys: slot B hands its (max, sum) to slot A, which merges both accumulators.
      // The buffer is rewritten only after slot B's last PV of a later unit, which the MMA
      // issues after slot A freed this unit's accumulators, i.e. after slot A's reads.
      float mB = -INFINITY, lB = 0.f;
      const bool split = !w.two && !w.dual && w.nt >= 2;   // the slots split the key tiles
      if (split) {
        if (x == 1) {
          merge_buf[row] = m_run;
          merge_buf[kBM + row] = l_run;
          warp_arrive(&bars[MERGE_FULL]);
        } else {
          ok = warp_wait<POLL>(&bars[MERGE_FULL], merges & 1, p.wait_ns);
          if (!ok) break;
          mB = merge_buf[row];
          lB = merge_buf[kBM + row];
        }
        ++merges;
      }
      if (w.two || w.dual || x == 0) {
        const bool valid = pr_u < w.urows;
        const int64_t prow = w.orow0 + pr_u;    // packed (query, head-in-group) row
        const int64_t qrow = prow / p.grp;      // the query's new row
        const int h = (w.g + (w.dual ? x : 0)) * p.grp + static_cast<int>(prow - qrow * p.grp);
        const float m = fmaxf(m_run, mB);
        const float ea = ex2_approx(m_run - m), eb = ex2_approx(mB - m);
        const float a = (l_run > 0.f) ? ea : 0.f;
        const float b = (lB > 0.f) ? eb : 0.f;
        const float lsum = a * l_run + b * lB;
        const float inv = 1.f / lsum;
        const float ca = a * inv, cb = b * inv;
        __nv_bfloat16* dst = p.out + (qrow * p.h_q + h) * D;
        // 32 output columns of this row from fp32 values: bf16, two 32-byte stores (four 16-byte
        // ones if the output is only 16-byte aligned).  A warp's rows lie h_q * d apart, so each
        // store instruction touches 32 lines: wider stores halve the instructions
        auto store32 = [&](int c0, const float (&f)[32]) {
          uint4 v4[4];
#pragma unroll
          for (int v = 0; v < 4; ++v)
            v4[v] = make_uint4(pack_bf16x2(f[8 * v + 0], f[8 * v + 1]), pack_bf16x2(f[8 * v + 2], f[8 * v + 3]),
                               pack_bf16x2(f[8 * v + 4], f[8 * v + 5]), pack_bf16x2(f[8 * v + 6], f[8 * v + 7]));
          uint4* d4 = reinterpret_cast<uint4*>(dst + c0);
          if (p.out_v8) {
            st_global_v8_pred(d4, v4[0], v4[1], valid);
            st_global_v8_pred(d4 + 2, v4[2], v4[3], valid);
          } else {
#pragma unroll
            for (int v = 0; v < 4; ++v) st_global_v4_pred(d4 + v, v4[v], valid);
          }
        };
        if (split) {
          // split keys: both accumulators, 64 columns at a time, each pair of loads one round trip
          // (warp-uniform; cb = 0 for a row slot B gave no weight)
#pragma unroll
          for (int hh = 0; hh < D / 64; ++hh) {
            uint32_t oa[64], ob[64];
            tmem_ld_x64_pair(tO + hh * 64, tOB + hh * 64, oa, ob);
#pragma unroll
            for (int q = 0; q < 2; ++q) {
              float f[32];
#pragma unroll
              for (int c = 0; c < 32; ++c)
                f[c] = fmaf(__uint_as_float(ob[32 * q + c]), cb, __uint_as_float(oa[32 * q + c]) * ca);
              store32(hh * 64 + q * 32, f);
            }
          }
        } else {
          // the whole accumulator row in one round trip
          uint32_t o[D];
          if constexpr (D == 128) tmem_ld_x128(tO, o);
          else tmem_ld_x64(tO, o);
#pragma unroll
          for (int ch = 0; ch < D / 32; ++ch) {
            float f[32];
#pragma unroll
            for (int c = 0; c < 32; ++c) f[c] = __uint_as_float(o[ch * 32 + c]) * ca;
            store32(ch * 32, f);
          }
        }
        if (p.lse) st_global_f32_pred(p.lse + qrow * p.h_q + h, (m + log2f(lsum)) * kLn2, valid);
        // this slot's O (and, with split keys, slot B's O too) may now be overwritten
        tc_fence_before_sync();
        warp_arrive(&bars[O_FREE + x]);
        if (!w.two && !w.dual) warp_arrive(&bars[O_FREE + 1]);
      }
    }
    if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
    tc_fence_before_sync();
  }
  __syncthreads();
  if (warp == 1) {
    tc_fence_after_sync();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* ptr = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
  });
  return fn;
}

// bf16 tensor [d3][d2][d1][d0] (d0 innermost) with box (64, b1, b2, b3), 128-byte swizzle.
bool make_map(CUtensorMap* m, const void* base, int rank, const uint64_t* dims, const uint32_t* box) {
  auto fn = encode_fn();
  if (!fn) return false;
  cuuint64_t gdim[4], gstride[3];
  cuuint32_t bdim[4], estr[4] = {1, 1, 1, 1};
  uint64_t stride = 2;
  for (int i = 0; i < rank; ++i) {
    gdim[i] = dims[i];
    bdim[i] = box[i];
    if (i > 0) gstride[i - 1] = stride;
    stride *= dims[i];
  }
  const CUresult r = fn(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, rank, const_cast<void*>(base), gdim, gstride, bdim,
                        estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                        CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  return r == CUDA_SUCCESS;
}

// The two launches of an attention call: the rotary/packing pre-pass and the forward.
constexpr int kPartBoth = 0, kPartRotate = 1, kPartCore = 2;

// Workspace of an attention call (byte offsets, each region 256-byte aligned): rotated
// queries, rotated new keys, the unit plan of a ragged batch (header, then up to
// max_pairs packed units) and, per new row, its problem's key bounds (16 bytes).
struct WsLayout {
  size_t khat, plan, row_bounds, total;
  int max_pairs;
};

WsLayout ws_layout(int64_t total_new, int32_t h_q, int32_t h_kv, int32_t d) {
  WsLayout l;
  const int64_t grp = h_q / std::max(h_kv, 1);
  l.max_pairs = static_cast<int>((total_new * grp + 2 * kBM - 1) / (2 * kBM));
  l.khat = align_up(static_cast<size_t>(total_new) * h_q * d * 2, 256);
  l.plan = l.khat + align_up(static_cast<size_t>(total_new) * h_kv * d * 2, 256);
  l.row_bounds = l.plan + align_up(sizeof(AttnPlanHdr) + static_cast<size_t>(l.max_pairs) * sizeof(AttnPlanUnit), 256);
  l.total = l.row_bounds + align_up(static_cast<size_t>(total_new) * sizeof(int4), 256);
  return l;
}

// One instantiation of the forward: the register split assumes the compiled register count
// (checked once), the dynamic shared memory is opted into once per device.
template <int D, bool PACKABLE, bool POLL, bool DUAL>
ssm_status launch_fwd_form(const AttnMaps& m, const AttnParams& p, int grid, cudaStream_t st) {
  using L = Layout<D>;
  static std::atomic<int> regs_ok{0};  // 0 unknown, 1 ok, 2 mismatch
  int st_regs = regs_ok.load();
  if (st_regs == 0) {
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, attn_fwd_kernel<D, PACKABLE, POLL, DUAL>) != cudaSuccess) return SSM_ERR_CUDA;
    st_regs = fa.numRegs == kLaunchRegs ? 1 : 2;
    regs_ok.store(st_regs);
  }
  if (st_regs != 1) return SSM_ERR_UNSUPPORTED;
  static std::atomic<uint64_t> attr_set{0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SSM_ERR_CUDA;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_set.load() & bit)) {
    if (cudaFuncSetAttribute(attn_fwd_kernel<D, PACKABLE, POLL, DUAL>, cudaFuncAttributeMaxDynamicSharedMemorySize, L::ALLOC) !=
        cudaSuccess)
      return SSM_ERR_CUDA;
    attr_set.fetch_or(bit);
  }
  ssm::launch_k(attn_fwd_kernel<D, PACKABLE, POLL, DUAL>, dim3(grid), dim3(kAttnThreads), L::ALLOC, st, m.q128, m.kc, m.vc,
                m.kn, m.vn, m.kc128, m.vc128, m.kn128, m.vn128, p);
  return launch_status();
}

// The forward for this call's wait limit: limits below the try_wait suspend window take the
// form whose waits poll without blocking (so that the limit holds); the usual limits, the
// form with blocking probes.
template <int D, bool PACKABLE>
ssm_status launch_fwd(const AttnMaps& m, const AttnParams& p, int grid, cudaStream_t st) {
  if (!PACKABLE && p.dual_heads) {
    if (p.wait_ns < kPollLimitNs) return launch_fwd_form<D, false, true, true>(m, p, grid, st);
    return launch_fwd_form<D, false, false, true>(m, p, grid, st);
  }
  if (p.wait_ns < kPollLimitNs) return launch_fwd_form<D, PACKABLE, true, false>(m, p, grid, st);
  return launch_fwd_form<D, PACKABLE, false, false>(m, p, grid, st);
}

template <int D>
ssm_status launch_attention(const void* q, const void* k_new, const void* v_new, const int32_t* pos,
                            const void* k_cache, const void* v_cache, bool uniform, int32_t batch_or_np,
                            int64_t new_rows_per_b, int64_t cache_rows_per_b, int32_t max_n_new,
                            int32_t max_n_cache, const ssm_attn_problem* problems, int32_t h_q, int32_t h_kv,
                            float rope_theta, float scale, void* out, float* lse, void* workspace,
                            cudaStream_t st, int part = kPartBoth) {
  using L = Layout<D>;
  const int grp = h_q / h_kv;
  const int64_t nb = uniform ? batch_or_np : 1;
  const int64_t total_new = uniform ? static_cast<int64_t>(batch_or_np) * new_rows_per_b : new_rows_per_b;
  const WsLayout wl = ws_layout(total_new, h_q, h_kv, D);
  auto* qhat = static_cast<__nv_bfloat16*>(workspace);
  auto* khat = reinterpret_cast<__nv_bfloat16*>(static_cast<uint8_t*>(workspace) + wl.khat);
  AttnMaps m;
  {
    const uint64_t dq[3] = {static_cast<uint64_t>(D),
                            static_cast<uint64_t>(uniform ? new_rows_per_b * grp : total_new * h_q),
                            static_cast<uint64_t>(uniform ? nb * h_kv : 1)};
    const uint32_t bq[3] = {64, kBM, 1};
    if (!make_map(&m.q128, qhat, 3, dq, bq)) return SSM_ERR_CUDA;
    const uint32_t bkv[4] = {64, 1, kSub, 1};
    const uint64_t dn[4] = {static_cast<uint64_t>(D), static_cast<uint64_t>(h_kv),
                            static_cast<uint64_t>(new_rows_per_b), static_cast<uint64_t>(nb)};
    if (!make_map(&m.kn, khat, 4, dn, bkv)) return SSM_ERR_CUDA;
    if (!make_map(&m.vn, v_new, 4, dn, bkv)) return SSM_ERR_CUDA;
    const uint32_t bkv128[4] = {64, 1, kBN, 1};
    if (!make_map(&m.kn128, khat, 4, dn, bkv128)) return SSM_ERR_CUDA;
    if (!make_map(&m.vn128, v_new, 4, dn, bkv128)) return SSM_ERR_CUDA;
    if (cache_rows_per_b > 0) {
      const uint64_t dc[4] = {static_cast<uint64_t>(D), static_cast<uint64_t>(h_kv),
                              static_cast<uint64_t>(cache_rows_per_b), static_cast<uint64_t>(nb)};
      if (!make_map(&m.kc, k_cache, 4, dc, bkv)) return SSM_ERR_CUDA;
      if (!make_map(&m.vc, v_cache, 4, dc, bkv)) return SSM_ERR_CUDA;
      if (!make_map(&m.kc128, k_cache, 4, dc, bkv128)) return SSM_ERR_CUDA;
      if (!make_map(&m.vc128, v_cache, 4, dc, bkv128)) return SSM_ERR_CUDA;
    } else {
      m.kc = m.kn;  // never read: no problem has cache rows
      m.vc = m.vn;
      m.kc128 = m.kn128;
      m.vc128 = m.vn128;
    }
  }
  AttnParams p{};
  p.problems = uniform ? nullptr : problems;
  p.n_new_u = uniform ? static_cast<int32_t>(new_rows_per_b) : 0;
  p.n_cache_u = uniform ? static_cast<int32_t>(cache_rows_per_b) : 0;
  p.h_q = h_q;
  p.h_kv = h_kv;
  p.grp = grp;
  p.new_rows_extent = static_cast<int32_t>(new_rows_per_b);
  p.qrows_g = uniform ? 0 : static_cast<int32_t>(total_new * grp);
  // Packed units need every problem to read one shared cache; a cache too small to hold two of
  // the longest prefixes (or no cache at all) is the only candidate.  Other batches run the
  // forward compiled without packed units, and the pre-pass makes no plan for them.
  const bool may_pack = !uniform && batch_or_np >= 2 &&
                        (cache_rows_per_b == 0 || 2 * static_cast<int64_t>(max_n_cache) > cache_rows_per_b);
  p.plan = may_pack ? reinterpret_cast<AttnPlanHdr*>(static_cast<uint8_t*>(workspace) + wl.plan) : nullptr;
  p.row_bounds = may_pack ? reinterpret_cast<int4*>(static_cast<uint8_t*>(workspace) + wl.row_bounds) : nullptr;
  p.scale_log2 = scale * kLog2e;
  p.out = static_cast<__nv_bfloat16*>(out);
  p.out_v8 = (reinterpret_cast<uintptr_t>(out) & 31u) == 0 ? 1 : 0;
  p.lse = lse;
  p.err = device_error_word();
  p.wait_ns = wait_limit_ns();
  const int n_prob = batch_or_np;
  if (part != kPartCore) {
    // persistent: as many CTAs per SM as fit (three at the kernel's register bound)
    static const int per_sm = resident_ctas(rope_pack_kernel<D>, kRopeWarps * 32, 0);
    const int64_t warps = static_cast<int64_t>(per_sm) * num_sms() * kRopeWarps;
    const int64_t rows = static_cast<int64_t>(n_prob) * max_n_new;
    // head parts per row: enough items for every warp when the batch has fewer rows than warps,
    // each part whole passes of kRopePasses x (32 / (D / 16)) head vectors
    const int pass_vecs = kRopePasses * (32 / (D / 16));
    const int n_pass = (h_q + h_kv + pass_vecs - 1) / pass_vecs;
    const int want = static_cast<int>(std::min<int64_t>((warps + rows - 1) / rows, n_pass));
    const int hper = ((n_pass + want - 1) / want) * pass_vecs;
    const int hsplit = (h_q + h_kv + hper - 1) / hper;
    const int64_t items = rows * hsplit;
    const int grid = static_cast<int>(std::min<int64_t>((items + kRopeWarps - 1) / kRopeWarps, warps / kRopeWarps));
    ssm::launch_k(rope_pack_kernel<D>, dim3(grid), dim3(kRopeWarps * 32), 0, st,
                  static_cast<const __nv_bfloat16*>(q), static_cast<const __nv_bfloat16*>(k_new), pos, p,
                  rope_freqs<D>(rope_theta), max_n_new, n_prob, wl.max_pairs, hsplit, hper, qhat, khat);
    const ssm_status s = launch_status();
    if (s != SSM_OK || part == kPartRotate) return s;
  }
  const int m_tiles = static_cast<int>((static_cast<int64_t>(max_n_new) * grp + kBM - 1) / kBM);
  // Problem units hold a pair of query tiles (both slots on every key tile) or, when that leaves
  // most SMs idle, single tiles (the slots split the key tiles and merge): the choice with the
  // shorter estimated makespan, in key tiles per slot chain, rounds of units x chain per unit
  // (a single tile's chain is half its key tiles plus about one tile for the merge).
  {
    const int64_t nt = ((static_cast<int64_t>(max_n_cache) + kSub - 1) / kSub +
                        (static_cast<int64_t>(max_n_new) + kSub - 1) / kSub + 3) / 4;
    const int64_t pgs = static_cast<int64_t>(n_prob) * h_kv;
    const int64_t sms = num_sms();
    const int64_t pair_cost = ((pgs * ((m_tiles + 1) / 2) + sms - 1) / sms) * nt;
    const int64_t single_cost = ((pgs * m_tiles + sms - 1) / sms) * ((nt + 1) / 2 + 1);
    p.tiles_per_unit = single_cost < pair_cost ? 1 : 2;
    // Problems of one query tile whose single-tile units take more than one round: units of two
    // kv heads (one tile each, each slot on its own head's key tiles) halve the unit count; a
    // unit's chain is then all its key tiles, both slots streaming at once.
    p.dual_heads = 0;
    if (!may_pack && m_tiles == 1 && h_kv % 2 == 0) {
      const int64_t dual_cost = ((pgs / 2 + sms - 1) / sms) * nt;
      if (dual_cost < single_cost) p.dual_heads = 1;
    }
  }
  p.units_per_pg = p.tiles_per_unit == 2 ? (m_tiles + 1) / 2 : m_tiles;
  const int64_t total_units =
      p.dual_heads ? static_cast<int64_t>(n_prob) * (h_kv / 2) : static_cast<int64_t>(p.units_per_pg) * n_prob * h_kv;
  if (total_units > INT32_MAX) return SSM_ERR_UNSUPPORTED;
  p.total_units = static_cast<int32_t>(total_units);
  if (!may_pack) return launch_fwd<D, false>(m, p, static_cast<int>(std::min<int64_t>(total_units, num_sms())), st);
  // packed units, if the pre-pass's plan chose them, number at most max_pairs per kv head
  const int64_t max_units = std::max<int64_t>(total_units, int64_t{wl.max_pairs} * h_kv);
  return launch_fwd<D, true>(m, p, static_cast<int>(std::min<int64_t>(max_units, num_sms())), st);
}

ssm_status check_attn(const void* q, const void* k_new, const void* v_new, const int32_t* pos,
                      int32_t h_q, int32_t h_kv, int32_t head_dim, float scale, float theta, void* out,
                      void* workspace) {
  if (!q || !k_new || !v_new || !pos || !out || !workspace) return SSM_ERR_INVALID_ARG;
  if (h_q <= 0 || h_kv <= 0) return SSM_ERR_INVALID_ARG;
  if (h_q % h_kv != 0) return SSM_ERR_SHAPE;
  if (head_dim != 64 && head_dim != 128) return SSM_ERR_UNSUPPORTED;
  if (!(scale > 0.f) || !(theta >= 0.f)) return SSM_ERR_INVALID_ARG;
  if (!aligned16(q) || !aligned16(k_new) || !aligned16(v_new) || !aligned16(out)) return SSM_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(workspace) & 255u) != 0) return SSM_ERR_INVALID_ARG;
  return SSM_OK;
}

}  // namespace
}  // namespace ssm

extern "C" {

size_t ssm_attention_workspace_size(int64_t total_new_rows, int32_t h_q, int32_t h_kv, int32_t head_dim) {
  if (total_new_rows <= 0 || h_q <= 0 || h_kv <= 0 || head_dim <= 0) return 0;
  return ssm::ws_layout(total_new_rows, h_q, h_kv, head_dim).total;
}

ssm_status ssm_attention(const void* q, const void* k_new, const void* v_new, const int32_t* pos,
                         const void* k_cache, const void* v_cache, int32_t batch, int32_t n_new,
                         int32_t n_cache, int32_t h_q, int32_t h_kv, int32_t head_dim,
                         float rope_theta, float scale, void* out, float* lse, void* workspace,
                         size_t ws_bytes, ssm_stream_t stream) {
  if (batch < 0 || n_new < 0 || n_cache < 0) return SSM_ERR_INVALID_ARG;
  if (batch == 0 || n_new == 0) return SSM_OK;
  ssm_status s = ssm::check_attn(q, k_new, v_new, pos, h_q, h_kv, head_dim, scale, rope_theta, out, workspace);
  if (s != SSM_OK) return s;
  if (n_cache > 0 && (!k_cache || !v_cache || !ssm::aligned16(k_cache) || !ssm::aligned16(v_cache)))
    return SSM_ERR_INVALID_ARG;
  if (ws_bytes < ssm_attention_workspace_size(static_cast<int64_t>(batch) * n_new, h_q, h_kv, head_dim))
    return SSM_ERR_CAPACITY;
  if (static_cast<int64_t>(batch) * h_kv > 65535) return SSM_ERR_UNSUPPORTED;
  if (static_cast<int64_t>(n_new) * (h_q / h_kv) > INT32_MAX / 2) return SSM_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (head_dim == 128)
    return ssm::launch_attention<128>(q, k_new, v_new, pos, k_cache, v_cache, true, batch, n_new, n_cache, n_new,
                                      n_cache, nullptr, h_q, h_kv, rope_theta, scale, out, lse, workspace, st);
  return ssm::launch_attention<64>(q, k_new, v_new, pos, k_cache, v_cache, true, batch, n_new, n_cache, n_new,
                                   n_cache, nullptr, h_q, h_kv, rope_theta, scale, out, lse, workspace, st);
}

static ssm_status attention_varlen_part(int part, const void* q, const void* k_new, const void* v_new,
                                const int32_t* pos, const void* k_cache, const void* v_cache,
                                int64_t total_new_rows, int64_t total_cache_rows,
                                const ssm_attn_problem* problems, int32_t n_problems,
                                int32_t max_n_new, int32_t max_n_cache, int32_t h_q,
                                int32_t h_kv, int32_t head_dim, float rope_theta, float scale,
                                void* out, float* lse, void* workspace, size_t ws_bytes,
                                ssm_stream_t stream) {
  if (n_problems < 0 || total_new_rows < 0 || total_cache_rows < 0 || max_n_new < 0 || max_n_cache < 0)
    return SSM_ERR_INVALID_ARG;
  if (n_problems == 0 || total_new_rows == 0 || max_n_new == 0) return SSM_OK;
  ssm_status s = ssm::check_attn(q, k_new, v_new, pos, h_q, h_kv, head_dim, scale, rope_theta, out, workspace);
  if (s != SSM_OK) return s;
  if (!problems) return SSM_ERR_INVALID_ARG;
  if (total_cache_rows > 0 && (!k_cache || !v_cache || !ssm::aligned16(k_cache) || !ssm::aligned16(v_cache)))
    return SSM_ERR_INVALID_ARG;
  if (ws_bytes < ssm_attention_workspace_size(total_new_rows, h_q, h_kv, head_dim)) return SSM_ERR_CAPACITY;
  if (static_cast<int64_t>(n_problems) * h_kv > 65535) return SSM_ERR_UNSUPPORTED;
  if (total_new_rows * h_q > INT32_MAX / 2 || total_cache_rows > INT32_MAX / 2) return SSM_ERR_UNSUPPORTED;
  cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
  if (head_dim == 128)
    return ssm::launch_attention<128>(q, k_new, v_new, pos, k_cache, v_cache, false, n_problems, total_new_rows,
                                      total_cache_rows, max_n_new, max_n_cache, problems, h_q, h_kv, rope_theta,
                                      scale, out, lse, workspace, st, part);
  return ssm::launch_attention<64>(q, k_new, v_new, pos, k_cache, v_cache, false, n_problems, total_new_rows,
                                   total_cache_rows, max_n_new, max_n_cache, problems, h_q, h_kv, rope_theta, scale,
                                   out, lse, workspace, st, part);
}


#define SSM_VARLEN_PARAMS                                                                                   \
  const void *q, const void *k_new, const void *v_new, const int32_t *pos, const void *k_cache,            \
      const void *v_cache, int64_t total_new_rows, int64_t total_cache_rows, const ssm_attn_problem *problems, \
      int32_t n_problems, int32_t max_n_new, int32_t max_n_cache, int32_t h_q, int32_t h_kv, int32_t head_dim, \
      float rope_theta, float scale, void *out, float *lse, void *workspace, size_t ws_bytes, ssm_stream_t stream
#define SSM_VARLEN_ARGS                                                                                     \
  q, k_new, v_new, pos, k_cache, v_cache, total_new_rows, total_cache_rows, problems, n_problems, max_n_new,  \
      max_n_cache, h_q, h_kv, head_dim, rope_theta, scale, out, lse, workspace, ws_bytes, stream

ssm_status ssm_attention_varlen(SSM_VARLEN_PARAMS) {
  return attention_varlen_part(ssm::kPartBoth, SSM_VARLEN_ARGS);
}

ssm_status ssm_attention_varlen_rotate(SSM_VARLEN_PARAMS) {
  return attention_varlen_part(ssm::kPartRotate, SSM_VARLEN_ARGS);
}

ssm_status ssm_attention_varlen_core(SSM_VARLEN_PARAMS) {
  return attention_varlen_part(ssm::kPartCore, SSM_VARLEN_ARGS);
}

}  // extern "C"
