// attn_common.cuh -- pieces of the attention forward (attention.cu): tile
// constants, the launch parameters, the per-problem geometry, key-tile validity
// and the warp-level barrier helpers.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cstdint>

#include "common.cuh"
#include "sm100_ptx.cuh"

namespace ssm {

constexpr int kBM = 128;            // query rows per tile (tcgen05 M) of the query-tile kernel
constexpr int kBN = 128;            // keys per tile
constexpr int kSub = 32;            // rows per TMA sub-box of a key tile
constexpr int kAttnThreads = 384;   // warpgroup 0: TMA Q/K (warp 0), MMA (warp 1), TMA V (warp 2), K/V watcher (warp 3); warpgroups 1, 2: slots A, B
// Register split: the kernels are launched with kLaunchRegs per thread (checked on the host);
// warpgroup 0 gives back down to kCtrlRegs and the two softmax warpgroups grow to
// kSoftmaxRegs: 128 * (168 - 72) = 256 * (216 - 168), so the split adds up exactly.
constexpr int kLaunchRegs = 168;
constexpr int kCtrlRegs = 72;
constexpr int kSoftmaxRegs = 216;
static_assert(128 * (kLaunchRegs - kCtrlRegs) >= 256 * (kSoftmaxRegs - kLaunchRegs), "register split");
static_assert(kAttnThreads * kLaunchRegs <= 65536, "launch registers");
constexpr int kPanel = 128 * 128;   // bytes of a 128-row x 64-column bf16 swizzle panel
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kLn2 = 0.6931471805599453f;
constexpr float kRescaleLog2 = 8.0f;  // rescale O only when a maximum grows by > 2^8
constexpr float kSpecSumMax = 65536.0f;  // a tile's row sum of p above this takes the exact path
constexpr uint32_t kTmemCols = 512;
constexpr uint64_t kDrainNs = 200000000ull;

// Packed units (ragged batches whose problems share one cache prefix and whose new rows
// follow one another): the rows of consecutive problems fill the query tiles together
// instead of each problem padding its own last tile.  A unit is a pair of 128-row tiles
// of one kv head's packed rows; its keys are the cache rows [0, c_max) followed by the
// new rows [nr_lo, nr_hi) of the problems it touches, and each row sees only its own
// problem's cache prefix and new rows.  The plan is made on the device by the RoPE
// pre-pass and read by the forward kernel.
struct AttnPlanHdr {
  int32_t packed;     // 1: the units below; 0: one problem per unit
  int32_t n_pairs;    // packed units per kv head
  int64_t cache_row;  // the shared cache's first row
  int64_t pad[2];
};
struct AttnPlanUnit {
  int32_t p0, rows;   // first packed row (query x head-in-group, within the kv head's block), rows (<= 256)
  int32_t c_max, pad; // cache keys: the largest prefix among the unit's problems
  int64_t nr_lo, nr_hi;  // new keys: the unit's problems' new rows
};

struct AttnParams {
  const ssm_attn_problem* problems;  // null: uniform batch
  int32_t n_new_u, n_cache_u;
  int32_t h_q, h_kv, grp;
  int32_t new_rows_extent;           // row extent of the new-K/V maps (OOB coordinate)
  int32_t qrows_g;                   // ragged batches: rotated query rows of one kv head (head-major layout)
  AttnPlanHdr* plan;                 // ragged batches: the unit plan (header, then units), else null
  int4* row_bounds;                  // ragged batches: per new row, its problem's (n_cache, new_row, new_row + n_new)
  int32_t units_per_pg;              // work units per (problem, kv head)
  int32_t tiles_per_unit;            // problem units: 128-row query tiles per unit (2: a pair, 1: single tiles)
  int32_t dual_heads;                // problem units of one query tile: two kv heads of one problem per unit
  int32_t total_units;
  float scale_log2;                  // softmax scale * log2(e)
  __nv_bfloat16* out;
  int32_t out_v8;                    // out is 32-byte aligned: 32-byte epilogue stores
  float* lse;
  unsigned* err;
  uint64_t wait_ns;
};

struct Geom {
  int64_t new_row, cache_row;
  int32_t n_new, n_cache;
};

__device__ __forceinline__ Geom problem_geom(const AttnParams& p, int prob) {
  Geom g;
  if (p.problems) {
    const ssm_attn_problem q = p.problems[prob];
    g.new_row = q.new_row;
    g.cache_row = q.cache_row;
    g.n_new = q.n_new;
    g.n_cache = q.n_cache;
  } else {
    g.n_new = p.n_new_u;
    g.n_cache = p.n_cache_u;
    g.new_row = static_cast<int64_t>(prob) * p.n_new_u;
    g.cache_row = 0;
  }
  return g;
}

__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi) {
  const __nv_bfloat162 h = __floats2bfloat162_rn(lo, hi);
  return *reinterpret_cast<const uint32_t*>(&h);
}

// This row's valid key range in each 32-row sub-box of key tile j of a packed unit: cache keys
// below the row's own prefix `lim`; new keys within the row's own problem, [nlo, nhi) counted from
// the unit's first new row.  The valid keys of a sub-box are columns [lo, hi); returns true if all
// 128 are valid.
__device__ __forceinline__ bool row_sub_bounds(int j, int n_csub, int n_nsub, int lim, int nlo, int nhi,
                                               int (&lo)[4], int (&hi)[4]) {
  bool full = true;
#pragma unroll
  for (int s4 = 0; s4 < 4; ++s4) {
    const int sub = 4 * j + s4;
    int a = 0, b = 0;
    if (sub < n_csub) {
      b = lim - sub * kSub;
    } else if (sub - n_csub < n_nsub) {
      const int kn = (sub - n_csub) * kSub;
      a = nlo - kn;
      b = nhi - kn;
    }
    a = min(max(a, 0), kSub);
    b = min(max(b, a), kSub);
    lo[s4] = a;
    hi[s4] = b;
    full = full && a == 0 && b == kSub;
  }
  return full;
}

// Valid keys in each 32-row sub-box of key tile j (cache sub-boxes first, then
// new-row sub-boxes); returns true if all 128 keys of the tile are valid.
__device__ __forceinline__ bool tile_valid_counts(int j, int n_csub, int n_nsub, const Geom& gm, int (&vcnt)[4]) {
  bool full = true;
#pragma unroll
  for (int s4 = 0; s4 < 4; ++s4) {
    const int sub = 4 * j + s4;
    int c;
    if (sub < n_csub) c = min(kSub, gm.n_cache - sub * kSub);
    else if (sub - n_csub < n_nsub) c = min(kSub, gm.n_new - (sub - n_csub) * kSub);
    else c = 0;
    vcnt[s4] = c;
    full = full && (c == kSub);
  }
  return full;
}

// Warp-level barrier use by the softmax warps.  Nothing here branches on the lane:
// tcgen05.ld/st are .sync.aligned, so the warp must still be one converged path when
// it reaches them, and a lane-0-only poll leaves lane 0 on a path of its own that
// warp-synchronous intrinsics (shuffles, __syncwarp) wait for but do not merge (a
// TMEM load issued that way ended a kernel with an unspecified launch failure).
// So every lane polls the barrier and the loop is steered by warp votes, and the
// single arrival of a warp is a predicated instruction rather than a branch.
// POLL: every probe is the non-blocking test_wait, so the limit is checked between probes
// whatever it is (a blocking try_wait may sleep until its phase completes, up to its ~20 us
// suspend window).  The host launches the polling form of a kernel only for wait limits
// below that window.
template <bool POLL = false>
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, uint64_t limit_ns) {
  if (__all_sync(0xffffffffu, mbar_test_wait(bar, parity))) return true;
  const uint64_t t0 = global_timer_ns();
  while (true) {
    if (__all_sync(0xffffffffu, POLL ? mbar_test_wait(bar, parity) : mbar_try_wait(bar, parity))) return true;
    if (__any_sync(0xffffffffu, global_timer_ns() - t0 > limit_ns)) return false;
  }
}

// Wait limits below this are polled (see warp_wait).
constexpr uint64_t kPollLimitNs = 20000;

__device__ __forceinline__ void warp_arrive(uint64_t* bar) {
  __syncwarp();
  mbar_arrive_if((threadIdx.x & 31) == 0, bar);
}

// The tensor maps the forward reads: queries packed by GQA group (128-row boxes),
// and the cache / new-row keys and values in 32-row and 128-row boxes.
struct AttnMaps {
  CUtensorMap q128, kc, vc, kn, vn, kc128, vc128, kn128, vn128;
};

}  // namespace ssm
