// suffix_geom.cuh -- closed-form description of the retained suffix set R_t
// (Sec. 3.2 "Suffix Region Partition" Eq. 1 and "Suffix Token Retention" Eqs. 2-5,
// with token budgets): membership of a position, the sizes of the three regions
// and the i-th retained position in ascending order.  Shared by the selector
// (select.cu) and the sparse-input gather that selects as it builds
// (build_input.cu).
#pragma once

#include <cstdint>

#include "ssm.h"

namespace ssm {

// Closed-form description of R_t for one configuration (shared by the host
// count and the device membership test).
struct SuffixGeom {
  int64_t s0;          // first suffix position
  int64_t end;         // one past the last generated position
  int64_t tail_start;  // first position of the tail block
  int64_t mid_first;   // start position of the first middle block
  int32_t B, L, M, T;
  int32_t n_sb;        // number of suffix blocks
  int32_t nm;          // number of middle blocks
  bool all_local;
};

__host__ __device__ inline SuffixGeom make_geom(const ssm_suffix_cfg& c) {
  SuffixGeom g{};
  const int32_t nb = c.gen_len / c.block_len;
  g.B = c.block_len;
  g.L = c.local_budget;
  g.M = c.middle_budget;
  g.T = c.tail_budget;
  g.s0 = static_cast<int64_t>(c.prompt_len) + static_cast<int64_t>(c.block_idx + 1) * c.block_len;
  g.end = static_cast<int64_t>(c.prompt_len) + c.gen_len;
  g.n_sb = nb - 1 - c.block_idx;
  g.tail_start = static_cast<int64_t>(c.prompt_len) + static_cast<int64_t>(nb - 1) * c.block_len;
  g.all_local = static_cast<int64_t>(g.n_sb) * g.B <= g.L;
  // middle blocks: suffix blocks other than the tail whose start is >= s0 + L
  const int64_t first = (static_cast<int64_t>(g.L) + g.B - 1) / g.B;  // blocks touched by local
  g.mid_first = g.s0 + first * g.B;
  const int64_t nm = static_cast<int64_t>(g.n_sb) - 1 - first;
  g.nm = nm > 0 ? static_cast<int32_t>(nm) : 0;
  return g;
}

// Is tail-block offset `o` one of the T evenly spaced offsets (j*(B-1))/(T-1)?
__host__ __device__ inline bool tail_keeps(const SuffixGeom& g, int64_t o) {
  if (g.T <= 0) return false;
  if (g.T >= g.B) return true;
  if (g.T == 1) return o == 0;
  const int64_t num = o * (g.T - 1);
  const int64_t j = (num + (g.B - 2)) / (g.B - 1);  // smallest j with j*(B-1)/(T-1) >= o
  return j <= g.T - 1 && (j * (g.B - 1)) / (g.T - 1) == o;
}

// Is middle block number `mi` (0-based among middle blocks) one of the kept ones?
__host__ __device__ inline bool middle_keeps(const SuffixGeom& g, int64_t mi) {
  if (g.nm <= g.M) return true;
  if (g.M <= 0) return false;
  const int64_t q = (mi * g.M + g.nm - 1) / g.nm;  // smallest q with q*nm/M >= mi
  return q < g.M && (q * g.nm) / g.M == mi;
}

__host__ __device__ inline bool keeps(const SuffixGeom& g, int64_t pos) {
  if (g.all_local) return true;
  if (pos < g.s0 + g.L) return true;                               // Eq. 2
  if (pos >= g.tail_start) return tail_keeps(g, pos - g.tail_start);  // Eq. 4
  if (pos >= g.mid_first && (pos - g.mid_first) % g.B == 0)         // Eq. 3
    return middle_keeps(g, (pos - g.mid_first) / g.B);
  return false;
}

// Region sizes of R_t: n_local, n_mid, and n_tail = tail tokens not already local (the three
// add up to |R_t|).  The tail offsets kept are j(B-1)/(T-1), j = 0..T-1 (all of them for
// T >= B, offset 0 for T = 1); those below the end of the local region are local already.
__host__ __device__ inline void region_counts(const SuffixGeom& g, int32_t& nl, int32_t& nmid, int32_t& nt) {
  if (g.n_sb <= 0) {
    nl = nmid = nt = 0;
    return;
  }
  if (g.all_local) {
    nl = g.n_sb * g.B;
    nmid = nt = 0;
    return;
  }
  nl = g.L;
  nmid = g.nm < g.M ? g.nm : g.M;
  const int64_t lo = g.s0 + g.L - g.tail_start;       // tail offsets below lo are local
  const int64_t first_o = lo > 0 ? lo : 0;
  if (g.T <= 0 || first_o >= g.B) {
    nt = 0;
  } else if (g.T >= g.B) {
    nt = static_cast<int32_t>(g.B - first_o);
  } else if (g.T == 1) {
    nt = first_o == 0 ? 1 : 0;
  } else {
    const int64_t j0 = (first_o * (g.T - 1) + (g.B - 2)) / (g.B - 1);  // first kept j with offset >= first_o
    nt = static_cast<int32_t>(g.T - j0 > 0 ? g.T - j0 : 0);
  }
}

// The i-th retained position of R_t in ascending order (0 <= i < nl + nmid + nt, the counts of
// region_counts): local tokens, then the kept middle blocks' start tokens, then the kept tail
// tokens past the local region.
__host__ __device__ inline int64_t retained_position(const SuffixGeom& g, int32_t nl, int32_t nmid, int64_t i) {
  if (i < nl) return g.s0 + i;                       // Eq. 2 (or every suffix token)
  i -= nl;
  if (i < nmid) {                                    // Eq. 3: block q*nm/M when nm > M
    const int64_t mi = g.nm <= g.M ? i : (i * g.nm) / g.M;
    return g.mid_first + mi * g.B;
  }
  i -= nmid;                                         // Eq. 4
  const int64_t lo = g.s0 + g.L - g.tail_start;
  const int64_t first_o = lo > 0 ? lo : 0;
  if (g.T >= g.B) return g.tail_start + first_o + i;
  if (g.T == 1) return g.tail_start;
  const int64_t j0 = (first_o * (g.T - 1) + (g.B - 2)) / (g.B - 1);
  return g.tail_start + ((j0 + i) * (g.B - 1)) / (g.T - 1);
}

}  // namespace ssm
