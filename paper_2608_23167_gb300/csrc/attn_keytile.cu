// attn_keytile.cu -- bidirectional attention (Sec. 1/2: non-causal DLM
// attention; Sec. 3.2: retained suffix tokens keep their rotary positions;
// Table 4 "PC.": prefix keys/values from a cache) for short query sets, with
// the keys on the tensor-memory lanes.
//
// A denoising step over a compacted sequence has few queries per head (the
// block plus the retained suffix: 32-172 rows at the paper's workloads) and
// many keys (the prefix).  With the queries on the M dimension of tcgen05.mma
// (128 rows per instruction) most of a second query tile would be padding; here
// the roles are swapped: S^T = K Q^T puts a 128-key tile on M and the queries
// of one (problem, kv head) on N, which only needs to be a multiple of 16.
// The softmax runs down the columns of S^T (one column per query), P^T goes
// to shared memory as the B operand of O^T += V^T P^T (V^T: the V tile read
// MN-major), and O^T accumulates in tensor memory with the head dimension on
// the lanes.
//
// One work unit = (problem, kv head), up to kKtMaxRows query rows (query x
// head-in-group, packed by rope_pack_kernel).  The two softmax warpgroups
// ("slots") either split the keys (rows <= kKtSplitKeysMax: both slots hold
// every query, slot A takes the even key tiles, slot B the odd ones, and the
// two partial softmax states are merged at the end) or split the queries (up
// to 96 each; both slots read every key tile).  Warp roles, the K/V rings, the
// K/V watcher and the carried barrier phases are those of attn_fwd_kernel in
// attention.cu.
//
// Softmax state per query column: a reference maximum m (log2 units, in shared
// memory, identical for every thread that holds the column) and a sum l, kept
// per thread over the thread's keys and reduced at the end of the unit.  A
// tile whose scores exceed m + 8 anywhere in the slot (one barrier-OR per
// tile) takes the slow path: exact column maxima across the slot's 128 keys,
// new m, O^T and l rescaled.  The first tile of a unit always takes it.
#include <cuda_bf16.h>

#include <atomic>

#include "attn_common.cuh"
#include "tmem_io.cuh"

namespace ssm {
namespace {

constexpr int kKtTile = 2 * kPanel;  // one 128-row x 128-column bf16 tile (head_dim 128)
constexpr int kKtStages = 2;         // stages of the K ring and of the V ring

enum KtBar {
  KT_Q_FULL = 0,
  KT_Q_EMPTY = 1,
  KT_K_FULL = 2,
  KT_K_EMPTY = KT_K_FULL + kKtStages,
  KT_V_FULL = KT_K_EMPTY + kKtStages,
  KT_V_EMPTY = KT_V_FULL + kKtStages,
  KT_S_FULL = KT_V_EMPTY + kKtStages,  // [2]: one per slot
  KT_P_FULL = KT_S_FULL + 2,           // [2]
  KT_O_DONE = KT_P_FULL + 2,           // [2]
  KT_O_FREE = KT_O_DONE + 2,           // [2]
  KT_DRAIN = KT_O_FREE + 2,
  KT_N_BARS = KT_DRAIN + 1
};

// Shared memory.  Region R (96 KB) holds Q and the two P^T buffers, laid out by
// the unit's mode:
//   queries split: Q in two 192-row panels (0, 24 KB; slot B's rows from row 96),
//                  P^T of slot x at 48 KB + 24 KB x (six 16-query panels);
//   keys split:    Q in two 128-row panels (0, 16 KB),
//                  P^T of slot x at 32 KB + 32 KB x (eight 16-query panels).
struct KtLayout {
  static constexpr int R = 0;
  static constexpr int K = 96 * 1024;
  static constexpr int V = K + kKtStages * kKtTile;
  static constexpr int MS = V + kKtStages * kKtTile;  // reference maxima m[2][128], fp32
  static constexpr int BAR = MS + 2 * 128 * 4;
  static constexpr int BYTES = BAR + KT_N_BARS * 8 + 8;
  static constexpr int ALLOC = BYTES + 1024;           // slack to align the base to 1024 B
  static_assert(ALLOC <= 232448, "shared memory budget");
};

__host__ __device__ constexpr int kt_qpanel(bool qs) { return qs ? 192 * 128 : 128 * 128; }
__host__ __device__ constexpr int kt_pt(bool qs, int x) { return qs ? 49152 + x * 24576 : 32768 + x * 32768; }

constexpr uint32_t kKtOCol = 256;  // O^T of slot x at 256 + 128 x; S^T (then nothing) at 128 x

struct KtUnit {
  Geom gm;
  int prob, g, rows, n_csub, n_nsub, nt, nA, nB;
  bool qs, valid;
};

__device__ __forceinline__ int round32(int v) { return (v + 31) & ~31; }

__device__ __forceinline__ KtUnit make_kt_unit(const AttnParams& p, int u) {
  KtUnit w;
  w.prob = u / p.h_kv;
  w.g = u - w.prob * p.h_kv;
  w.gm = problem_geom(p, w.prob);
  w.rows = w.gm.n_new * p.grp;
  // the host guarantees rows <= kKtMaxRows (max_n_new * grp); a table entry
  // beyond it is skipped (and reported by the MMA thread)
  w.valid = w.rows > 0 && w.rows <= kKtMaxRows;
  w.qs = w.rows > kKtSplitKeysMax;
  // slot widths (the MMA N and the softmax columns) are multiples of 32, so the
  // softmax works on whole 32-column chunks
  if (w.qs) {
    w.nA = round32((w.rows + 1) / 2);
    w.nB = round32(w.rows - w.nA);
  } else {
    w.nA = w.nB = round32(w.rows);
  }
  w.n_csub = (w.gm.n_cache + kSub - 1) / kSub;
  w.n_nsub = (w.gm.n_new + kSub - 1) / kSub;
  w.nt = (w.n_csub + w.n_nsub + 3) / 4;
  return w;
}

// A softmax thread holds, per 32-column chunk of S^T (two tcgen05.ld.16x256b.x4
// blocks), 4 keys x 8 columns: keys (TMEM lanes) 32 quarter + lane / 4 + 8 kb,
// columns 32 ch + 8 gq + 2 (lane % 4) + c for gq = 0..3, c = 0, 1.  Register
// index of (kb, gq, c) within the chunk:
__host__ __device__ constexpr int CI(int kb, int gq, int c) { return 16 * (kb >> 1) + 4 * gq + 2 * (kb & 1) + c; }
// ... and index of the thread's column (gq, c) of chunk ch among its 32 columns:
__host__ __device__ constexpr int JC(int ch, int gq, int c) { return 8 * ch + 2 * gq + c; }

// Loads chunk ch of this warp's S^T (or O^T) fragment; keys that are not valid
// (kv false, only in a tile that straddles a segment end) read as -inf.
__device__ __forceinline__ void kt_chunk(uint32_t t0, uint32_t t1, int ch, bool full, const bool (&kv)[4],
                                         float (&r)[32]) {
  uint32_t u[32];
  tmem_ld_16x256b_pair(t0 + 32 * ch, t1 + 32 * ch, u);
#pragma unroll
  for (int i = 0; i < 32; ++i) r[i] = __uint_as_float(u[i]);
  if (!full) {
#pragma unroll
    for (int kb = 0; kb < 4; ++kb)
      if (!kv[kb])
#pragma unroll
        for (int gq = 0; gq < 4; ++gq) {
          r[CI(kb, gq, 0)] = -INFINITY;
          r[CI(kb, gq, 1)] = -INFINITY;
        }
  }
}

__global__ void __launch_bounds__(kAttnThreads, 1) attn_keytile_kernel(
    const __grid_constant__ CUtensorMap tm_q128, const __grid_constant__ CUtensorMap tm_q96,
    const __grid_constant__ CUtensorMap tm_kc, const __grid_constant__ CUtensorMap tm_vc,
    const __grid_constant__ CUtensorMap tm_kn, const __grid_constant__ CUtensorMap tm_vn,
    const __grid_constant__ CUtensorMap tm_kc128, const __grid_constant__ CUtensorMap tm_vc128,
    const __grid_constant__ CUtensorMap tm_kn128, const __grid_constant__ CUtensorMap tm_vn128,
    const AttnParams p) {
  using L = KtLayout;
  constexpr int D = 128;

  extern __shared__ uint8_t smem_raw[];
  // aligned by pointer arithmetic on the shared array, so accesses through it stay shared-memory accesses
  uint8_t* smem = smem_raw + ((1024u - (smem_u32(smem_raw) & 1023u)) & 1023u);
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + L::BAR);
  uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + KT_N_BARS);
  float* m_all = reinterpret_cast<float*>(smem + L::MS);  // -m per column, [2][128]

  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const bool uniform = p.problems == nullptr;

  // No control flow here depends on the lane: each control warp walks its loop as one
  // converged path and lane 0 issues through predicated instructions (the *_if helpers).
  const bool leader = lane == 0;
  if (warp == 0) {
    mbar_init_if(leader, &bars[KT_Q_FULL], 1);
    mbar_init_if(leader, &bars[KT_Q_EMPTY], 1);
    for (int s = 0; s < kKtStages; ++s) {
      mbar_init_if(leader, &bars[KT_K_FULL + s], 1);
      mbar_init_if(leader, &bars[KT_K_EMPTY + s], 1);
      mbar_init_if(leader, &bars[KT_V_FULL + s], 1);
      mbar_init_if(leader, &bars[KT_V_EMPTY + s], 1);
    }
    for (int x = 0; x < 2; ++x) {
      mbar_init_if(leader, &bars[KT_S_FULL + x], 1);
      mbar_init_if(leader, &bars[KT_P_FULL + x], 5);  // one arrival per softmax warp, one from the K/V watcher
      mbar_init_if(leader, &bars[KT_O_DONE + x], 1);
      mbar_init_if(leader, &bars[KT_O_FREE + x], 4);
    }
    mbar_init_if(leader, &bars[KT_DRAIN], 1);
    fence_mbar_init();
  }
  if (warp == 1) {
    tmem_alloc(tmem_slot, kTmemCols);
    tmem_relinquish_alloc_permit();
  }
  if (warp == 0) {
    tma_prefetch_desc(&tm_q128);
    tma_prefetch_desc(&tm_q96);
    tma_prefetch_desc(&tm_kc);
    tma_prefetch_desc(&tm_vc);
    tma_prefetch_desc(&tm_kn);
    tma_prefetch_desc(&tm_vn);
  }
  tc_fence_before_sync();
  __syncthreads();
  tc_fence_after_sync();
  const uint32_t tmem = *tmem_slot;

  if (warp < 4) {
    setmaxnreg_dec<kCtrlRegs>();
    if (warp == 0 || warp == 2) {
      // ------------------------------------------------------------- TMA producers
      // warp 0 loads Q and the K ring, warp 2 the V ring, each at its own pace
      const int half = warp == 2 ? 1 : 0;
      bool ok = true;
      int qcount = 0;  // units whose Q was loaded
      int fills = 0;   // tiles loaded into this ring so far (all units)
      for (int u = blockIdx.x; u < p.total_units && ok; u += gridDim.x) {
        const KtUnit w = make_kt_unit(p, u);
        if (!w.valid) continue;
        if (!half) {
          if (qcount > 0) ok = warp_wait(&bars[KT_Q_EMPTY], (qcount - 1) & 1, p.wait_ns);
          if (!ok) break;
          int qy, qz;
          if (uniform) {
            qy = 0;
            qz = w.prob * p.h_kv + w.g;
          } else {
            qy = static_cast<int>(static_cast<int64_t>(w.g) * p.qrows_g + w.gm.new_row * p.grp);
            qz = 0;
          }
          if (w.qs) {
            // slot A's rows [0, nA) at panel row 0, slot B's [nA, rows) at panel row 96
            mbar_arrive_expect_tx_if(leader, &bars[KT_Q_FULL], 2 * 2 * 96 * 128);
#pragma unroll
            for (int x = 0; x < 2; ++x)
#pragma unroll
              for (int pn = 0; pn < 2; ++pn)
                tma_load_3d_if(leader, smem + L::R + pn * kt_qpanel(true) + x * 96 * 128, &tm_q96, &bars[KT_Q_FULL], pn * 64,
                            qy + x * w.nA, qz);
          } else {
            mbar_arrive_expect_tx_if(leader, &bars[KT_Q_FULL], 2 * 128 * 128);
#pragma unroll
            for (int pn = 0; pn < 2; ++pn)
              tma_load_3d_if(leader, smem + L::R + pn * kt_qpanel(false), &tm_q128, &bars[KT_Q_FULL], pn * 64, qy, qz);
          }
          ++qcount;
        }
        const int c3 = uniform ? w.prob : 0;
        for (int jt = 0; jt < w.nt && ok; ++jt) {
          const int st = fills % kKtStages, fill = fills / kKtStages;
          if (fill > 0) ok = warp_wait(&bars[(half ? KT_V_EMPTY : KT_K_EMPTY) + st], (fill - 1) & 1, p.wait_ns);
          if (!ok) break;
          uint64_t* full = &bars[(half ? KT_V_FULL : KT_K_FULL) + st];
          mbar_arrive_expect_tx_if(leader, full, kKtTile);
          uint8_t* dst = smem + (half ? L::V : L::K) + st * kKtTile;
          const int sub0 = 4 * jt;
          const bool whole_cache = sub0 + 3 < w.n_csub && (sub0 + 4) * kSub <= w.gm.n_cache;
          const bool whole_new = sub0 >= w.n_csub && (sub0 - w.n_csub + 4) * kSub <= w.gm.n_new;
          if (whole_cache || whole_new) {
            const CUtensorMap* map = whole_cache ? (half ? &tm_vc128 : &tm_kc128) : (half ? &tm_vn128 : &tm_kn128);
            const int c2 = whole_cache ? (uniform ? sub0 * kSub : static_cast<int>(w.gm.cache_row + sub0 * kSub))
                                       : (uniform ? (sub0 - w.n_csub) * kSub
                                                  : static_cast<int>(w.gm.new_row + (sub0 - w.n_csub) * kSub));
#pragma unroll
            for (int pn = 0; pn < 2; ++pn) tma_load_4d_if(leader, dst + pn * kPanel, map, full, pn * 64, w.g, c2, c3);
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
              for (int pn = 0; pn < 2; ++pn)
                tma_load_4d_if(leader, dst + pn * kPanel + sb * kSub * 128, map, full, pn * 64, w.g, c2, c3);
            }
          }
          ++fills;
        }
      }
      if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
      // every copy in flight lands before the CTA's shared memory is released, on every path
      // (a consumer that timed out may have left this warp's last fills unconsumed)
      if (!half && qcount > 0) warp_wait(&bars[KT_Q_FULL], (qcount - 1) & 1, kDrainNs);
      for (int i = max(0, fills - kKtStages); i < fills; ++i)
        warp_wait(&bars[(half ? KT_V_FULL : KT_K_FULL) + i % kKtStages], (i / kKtStages) & 1, kDrainNs);
    } else if (warp == 1) {
      // ------------------------------------------------------------- MMA issuer
      bool ok = true;
      const uint32_t sK = smem_u32(smem + L::K), sV = smem_u32(smem + L::V), sR = smem_u32(smem + L::R);
      int ucount = 0;            // units processed
      int kbase = 0, vbase = 0;  // global index of the unit's first K / V tile
      int pv0 = 0, pv1 = 0;      // PV GEMMs issued per slot (all units)
      for (int u = blockIdx.x; u < p.total_units && ok; u += gridDim.x) {
        const KtUnit w = make_kt_unit(p, u);
        if (!w.valid) {
          if (w.rows > kKtMaxRows) record_error(p.err, SSM_ERR_SHAPE);
          continue;
        }
        ok = warp_wait(&bars[KT_Q_FULL], ucount & 1, p.wait_ns);
        if (!ok) break;
        const bool qs = w.qs;
        uint32_t id_qk[2], id_pv[2], qb[2], pb[2];
#pragma unroll
        for (int x = 0; x < 2; ++x) {
          const int n = x ? w.nB : w.nA;
          id_qk[x] = idesc_bf16_f32(128, n, false, false);  // S^T = K Q^T: both K-major
          id_pv[x] = idesc_bf16_f32(128, n, true, true);    // O^T += V^T P^T: both MN-major
          qb[x] = sR + (qs ? x * 96 * 128 : 0);
          pb[x] = sR + kt_pt(qs, x);
        }
        const int qpan = kt_qpanel(qs);
        int kx0 = 0, kx1 = 0;        // jobs issued per slot in this unit
        int jlast0 = 0, jlast1 = 0;  // key tile of each slot's latest S^T
        bool freed0 = false, freed1 = false;
        // one O_FREE wait per slot and unit: the previous unit's epilogue has read this slot's O^T
        auto wait_o_free = [&](int x) -> bool {
          bool& f = x ? freed1 : freed0;
          if (f) return true;
          f = true;
          return ucount == 0 || warp_wait(&bars[KT_O_FREE + x], (ucount - 1) & 1, p.wait_ns);
        };
        // O^T_X += V^T(j) P^T_X for slot X's latest job
        auto issue_pv = [&](int x) -> bool {
          const int jp = x ? jlast1 : jlast0, k = (x ? kx1 : kx0) - 1;
          int& pv = x ? pv1 : pv0;
          if (!wait_o_free(x)) return false;
          // the K/V watcher's share of this phase vouches for V(jp) and this slot's next K tile
          if (!warp_wait(&bars[KT_P_FULL + x], pv & 1, p.wait_ns)) return false;
          const int vi = vbase + jp;
          tc_fence_after_sync();
          const uint32_t vaddr = sV + (vi % kKtStages) * kKtTile;
          const uint32_t d_tmem = tmem + kKtOCol + x * 128;
#pragma unroll
          for (int kk = 0; kk < kBN / 16; ++kk)
            umma_bf16_ss_if(leader, d_tmem, sdesc_sw128(vaddr + kk * 16 * 128, kPanel, 1024),
                         sdesc_sw32(pb[x] + kk * 16 * 32, 4096, 256), id_pv[x], (kk > 0 || k > 0) ? 1u : 0u);
          umma_commit_if(leader, &bars[KT_O_DONE + x]);
          if (!qs || x == 1) umma_commit_if(leader, &bars[KT_V_EMPTY + vi % kKtStages]);
          ++pv;
          return true;
        };
        const int n_jobs = qs ? 2 * w.nt : w.nt;
        for (int t = 0; t < n_jobs && ok; ++t) {
          const int x = t & 1;
          const int j = qs ? (t >> 1) : t;
          const int ki = kbase + j;
          if ((x ? kx1 : kx0) > 0)
            ok = issue_pv(x);  // the watcher's share of P_FULL vouches for this slot's next K tile too
          else
            ok = warp_wait(&bars[KT_K_FULL + ki % kKtStages], (ki / kKtStages) & 1, p.wait_ns);
          if (!ok) break;
          const uint32_t kaddr = sK + (ki % kKtStages) * kKtTile;
          const uint32_t s_tmem = tmem + x * 128;
#pragma unroll
          for (int kk = 0; kk < D / 16; ++kk) {
            const uint32_t off = (kk >> 2) * kPanel + (kk & 3) * 32;
            const uint32_t qoff = (kk >> 2) * qpan + (kk & 3) * 32;
            umma_bf16_ss_if(leader, s_tmem, sdesc_sw128(kaddr + off, 16, 1024), sdesc_sw128(qb[x] + qoff, 16, 1024), id_qk[x],
                         kk > 0 ? 1u : 0u);
          }
          umma_commit_if(leader, &bars[KT_S_FULL + x]);
          if (!qs || x == 1) umma_commit_if(leader, &bars[KT_K_EMPTY + ki % kKtStages]);
          if (x) {
            jlast1 = j;
            ++kx1;
          } else {
            jlast0 = j;
            ++kx0;
          }
        }
        // The next unit's Q is loaded once Q_EMPTY completes.  After a keys-split unit
        // whose successor splits the queries, that Q overlaps this unit's P^T of slot A,
        // so Q_EMPTY then waits for the final PV GEMMs too.
        bool gate = false;
        if (!qs) {
          for (int u2 = u + gridDim.x; u2 < p.total_units; u2 += gridDim.x) {
            const KtUnit w2 = make_kt_unit(p, u2);
            if (w2.valid) {
              gate = w2.qs;
              break;
            }
          }
        }
        if (ok && !gate) umma_commit_if(leader, &bars[KT_Q_EMPTY]);
        if (ok && kx0 > 0) ok = issue_pv(0);
        if (ok && kx1 > 0) ok = issue_pv(1);
        if (ok && gate) umma_commit_if(leader, &bars[KT_Q_EMPTY]);
        if (ok) ok = wait_o_free(0) && wait_o_free(1);
        kbase += w.nt;
        vbase += w.nt;
        ++ucount;
      }
      if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
      // every issued MMA completes before tensor memory is released
      umma_commit_if(leader, &bars[KT_DRAIN]);
      warp_wait(&bars[KT_DRAIN], 0, kDrainNs);
    } else {
      // ------------------------------------------------------------- K/V watcher (warp 3)
      // Takes the K and V waits off the MMA warp (each mbarrier test costs it issue time):
      // for each PV it waits until that PV's V tile and the K tile of the slot's next S^T
      // have landed, then adds its arrival to the slot's P_FULL phase, after seeing the
      // slot's previous phase complete.  V tiles are confirmed in ring order; for K the
      // fill before the awaited one is known from the slot's S^T completions, observed in
      // order (the same scheme as attn_fwd_kernel).
      bool ok = true;
      int kbase = 0;
      int done0 = 0, done1 = 0;
      int vconf = 0;  // V tiles (all units) confirmed landed, in order
      auto vouch = [&](int x, int jp, int jk) -> bool {
        int& d = x ? done1 : done0;
        if (d > 0 && !warp_wait(&bars[KT_P_FULL + x], (d - 1) & 1, p.wait_ns)) return false;
        // slot x's d-th QK^T (on K tile jp) has completed, so tile jp has landed; every S
        // of each slot is seen here in order, so the fill before any K tile waited for
        // below is known to have landed (split keys: tile jp itself; both slots on every
        // tile: tile jp - 1, or the previous unit's last tile), and the fill after it
        // needs this vouch: each parity wait stays within its two-phase window
        if (!warp_wait(&bars[KT_S_FULL + x], d & 1, p.wait_ns)) return false;
        for (; vconf <= kbase + jp; ++vconf)
          if (!warp_wait(&bars[KT_V_FULL + vconf % kKtStages], (vconf / kKtStages) & 1, p.wait_ns)) return false;
        if (jk >= 0) {
          const int ki = kbase + jk;
          if (!warp_wait(&bars[KT_K_FULL + ki % kKtStages], (ki / kKtStages) & 1, p.wait_ns)) return false;
        }
        mbar_arrive_if(leader, &bars[KT_P_FULL + x]);
        ++d;
        return true;
      };
      for (int u = blockIdx.x; u < p.total_units && ok; u += gridDim.x) {
        const KtUnit w = make_kt_unit(p, u);
        if (!w.valid) continue;
        int kx0 = 0, kx1 = 0, jlast0 = 0, jlast1 = 0;
        const int n_jobs = w.qs ? 2 * w.nt : w.nt;
        for (int t = 0; t < n_jobs && ok; ++t) {
          const int x = t & 1;
          const int j = w.qs ? (t >> 1) : t;
          if ((x ? kx1 : kx0) > 0) ok = vouch(x, x ? jlast1 : jlast0, j);
          if (x) {
            jlast1 = j;
            ++kx1;
          } else {
            jlast0 = j;
            ++kx0;
          }
        }
        if (ok && kx0 > 0) ok = vouch(0, jlast0, -1);
        if (ok && kx1 > 0) ok = vouch(1, jlast1, -1);
        kbase += w.nt;
      }
      if (!ok) record_error(p.err, SSM_ERR_TIMEOUT);
    }
  } else {
    // ------------------------------------------------------------- softmax slots (warps 4..11)
    setmaxnreg_inc<kSoftmaxRegs>();
    const int x = (warp - 4) >> 2;  // slot
    const int quarter = warp & 3;   // TMEM lanes 32 * quarter .. + 31 belong to this warp
    const uint32_t bar_id = 1 + x;  // named barrier of this slot's 128 threads; 3 = both slots
    const uint32_t lane_off = static_cast<uint32_t>(quarter * 32) << 16;
    const uint32_t tS0 = tmem + lane_off + x * 128, tS1 = tS0 + (16u << 16);
    const uint32_t tO0 = tmem + lane_off + kKtOCol + x * 128, tO1 = tO0 + (16u << 16);
    const uint32_t tOA = tmem + lane_off + kKtOCol, tOB = tOA + 128;  // 32x32b views for the epilogue
    float* nm_s = m_all + x * 128;  // -m per column of this slot
    const int cpair = 2 * (lane & 3);  // this thread's first column of each 8-column group
    const int krow0 = lane >> 2;       // key rows 32 quarter + krow0 + 8 kb
    const uint32_t sw = (lane >> 4) & 1;  // 32-byte swizzle: bit 2 of the key row
    const float sc = p.scale_log2;
    // A wait that expires clears ok; the warp then skips its remaining waits but keeps
    // the same control flow, so the slot's named barriers never miss a participant.
    bool ok = true;
    int sj = 0;  // S^T tiles consumed by this slot (all units)
    for (int u = blockIdx.x; u < p.total_units; u += gridDim.x) {
      const KtUnit w = make_kt_unit(p, u);
      if (!w.valid) continue;
      const bool qs = w.qs;
      const int jobs = qs ? w.nt : (x == 0 ? (w.nt + 1) / 2 : w.nt / 2);
      const int n = x ? w.nB : w.nA;  // columns of this slot (a multiple of 32)
      const int nch = n >> 5;
      uint8_t* pt = smem + L::R + kt_pt(qs, x);
      // this thread's P^T words: key row 32 quarter + krow0 (+ 8 kb), the 4-byte pair of lane % 4 in
      // the row's 16-byte half (g % 2) ^ sw of 16-query panel g / 2
      uint8_t* pt_row = pt + (quarter * 32 + krow0) * 32 + (lane & 3) * 4;
      uint8_t* pt_even = pt_row + (sw << 4);
      uint8_t* pt_odd = pt_row + ((sw ^ 1u) << 4);
      // per column of this thread: the sum over its keys; -m (the reference maximum, log2
      // units) of every column of the slot lives in shared memory (nm_s), written in the
      // slow path by the lanes that hold each column in warp quarter 0
      float l[32];
#pragma unroll
      for (int i = 0; i < 32; ++i) l[i] = 0.f;
      for (int k = 0; k < jobs; ++k) {
        const int j = qs ? k : 2 * k + x;
        if (ok) ok = warp_wait(&bars[KT_S_FULL + x], sj & 1, p.wait_ns);
        tc_fence_after_sync();
        int vcnt[4];
        const bool full = tile_valid_counts(j, w.n_csub, w.n_nsub, w.gm, vcnt);
        // valid keys of this warp's 32-row sub-box (sub-box = TMEM lane quarter)
        const int sub = 4 * j + quarter;
        const int myc = sub < w.n_csub ? min(kSub, w.gm.n_cache - sub * kSub)
                                       : (sub - w.n_csub < w.n_nsub ? min(kSub, w.gm.n_new - (sub - w.n_csub) * kSub) : 0);
        bool kv[4];
#pragma unroll
        for (int kb = 0; kb < 4; ++kb) kv[kb] = krow0 + 8 * kb < myc;
        const bool first = k == 0;
        // pass: p = 2^(s * scale * log2 e - m) for every chunk, P^T (bf16 pairs) to shared
        // memory, the column sums added to l (scaled by addf in a redo); returns the largest
        // exponent.  Chunk ch + 1 is loaded while chunk ch is processed.
        auto exp_pass = [&](bool redo, uint32_t addf) -> float {
          float mx[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
          uint32_t ua[32], ub[32];
          tmem_ld_16x256b_pair_issue(tS0, tS1, ua);
#pragma unroll
          for (int ch = 0; ch < 4; ++ch) {
            if (ch < nch) {
              // -m of the chunk's columns (read while the chunk's load is in flight)
              float2 nmv[4];
#pragma unroll
              for (int gq = 0; gq < 4; ++gq) nmv[gq] = *reinterpret_cast<const float2*>(nm_s + 32 * ch + 8 * gq + cpair);
              uint32_t(&u)[32] = (ch & 1) ? ub : ua;
              tmem_wait_ld_32(u);
              if (ch + 1 < nch) tmem_ld_16x256b_pair_issue(tS0 + 32 * (ch + 1), tS1 + 32 * (ch + 1), (ch & 1) ? ua : ub);
              float r[32];
#pragma unroll
              for (int i = 0; i < 32; ++i) r[i] = __uint_as_float(u[i]);
              if (!full) {  // per-lane selects, no branch: the warp stays converged
#pragma unroll
                for (int kb = 0; kb < 4; ++kb)
#pragma unroll
                  for (int gq = 0; gq < 4; ++gq) {
                    r[CI(kb, gq, 0)] = kv[kb] ? r[CI(kb, gq, 0)] : -INFINITY;
                    r[CI(kb, gq, 1)] = kv[kb] ? r[CI(kb, gq, 1)] : -INFINITY;
                  }
              }
#pragma unroll
              for (int gq = 0; gq < 4; ++gq) {
                const int g = 4 * ch + gq;
                uint32_t* prow = reinterpret_cast<uint32_t*>(((g & 1) ? pt_odd : pt_even) + (g >> 1) * 4096);
                float p[8];
#pragma unroll
                for (int kb = 0; kb < 4; ++kb) {
                  float x0, x1;
                  ffma2(x0, x1, r[CI(kb, gq, 0)], r[CI(kb, gq, 1)], sc, sc, nmv[gq].x, nmv[gq].y);
                  if (!redo) mx[kb] = fmax3(mx[kb], x0, x1);
                  p[2 * kb] = ex2_approx(x0);
                  p[2 * kb + 1] = ex2_approx(x1);
                  prow[kb * 64] = pack_bf16x2(p[2 * kb], p[2 * kb + 1]);  // key row + 8 kb: 256 bytes on
                }
                float a0 = p[0], a1 = p[1], b0 = p[4], b1 = p[5];
                fadd2_acc(a0, a1, p[2], p[3]);
                fadd2_acc(b0, b1, p[6], p[7]);
                fadd2_acc(a0, a1, b0, b1);
                if (redo) {
                  a0 = ((addf >> JC(ch, gq, 0)) & 1u) ? a0 : 0.f;
                  a1 = ((addf >> JC(ch, gq, 1)) & 1u) ? a1 : 0.f;
                }
                fadd2_acc(l[JC(ch, gq, 0)], l[JC(ch, gq, 1)], a0, a1);
              }
            }
          }
          return fmaxf(fmaxf(mx[0], mx[1]), fmaxf(mx[2], mx[3]));
        };
        uint32_t addf = 0xffffffffu;  // columns whose redo sums are added to l
        // Speculative pass against the current reference (not on a unit's first tile, which
        // has none); then one OR across the slot: did any exponent exceed 8?
        bool need = first;
        if (!first) need = named_barrier_or(bar_id, 128, exp_pass(false, addf) > kRescaleLog2);
        if (need) {
          // ---- slow path: exact column maxima over the tile's keys, new m; the speculative
          // sums already in l become exact by the same factor alpha as O^T (p_old * alpha =
          // p_new), except where the maximum jumped by >= 100 (2^x may have overflowed there:
          // l restarts from this tile's sums, earlier terms being below 2^-80 of them)
          float cm[32];
#pragma unroll
          for (int i = 0; i < 32; ++i) cm[i] = -INFINITY;
#pragma unroll
          for (int ch = 0; ch < 4; ++ch) {
            if (ch < nch) {
              float r[32];
              kt_chunk(tS0, tS1, ch, full, kv, r);
#pragma unroll
              for (int gq = 0; gq < 4; ++gq) {
                const float2 nmv = first ? make_float2(0.f, 0.f)
                                         : *reinterpret_cast<const float2*>(nm_s + 32 * ch + 8 * gq + cpair);
#pragma unroll
                for (int kb = 0; kb < 4; ++kb) {
                  float x0, x1;  // scores against the current reference (against 0 on the first tile)
                  ffma2(x0, x1, r[CI(kb, gq, 0)], r[CI(kb, gq, 1)], sc, sc, nmv.x, nmv.y);
                  cm[JC(ch, gq, 0)] = fmaxf(cm[JC(ch, gq, 0)], x0);
                  cm[JC(ch, gq, 1)] = fmaxf(cm[JC(ch, gq, 1)], x1);
                }
              }
            }
          }
          // lanes with the same lane % 4 hold the same columns
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            if ((i >> 3) < nch) {
              float v = cm[i];
              v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 4));
              v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 8));
              v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, 16));
              cm[i] = v;
            }
          }
          // across the slot's four warps through the first 2 KB of this slot's P^T buffer:
          // the P^T rewritten below replaces it, and the OR above (on a unit's first tile:
          // the slot's previous PV, complete before this S^T tile was committed) orders the
          // scratch after every earlier use of the buffer
          float* scr = reinterpret_cast<float*>(pt);  // [4][128]
#pragma unroll
          for (int ch = 0; ch < 4; ++ch)
            if (ch < nch)
#pragma unroll
              for (int gq = 0; gq < 4; ++gq)
                st_shared_f32x2_if(lane < 4, scr + quarter * 128 + 32 * ch + 8 * gq + cpair, cm[JC(ch, gq, 0)],
                                   cm[JC(ch, gq, 1)]);
          named_barrier_sync(bar_id, 128);
#pragma unroll
          for (int ch = 0; ch < 4; ++ch) {
            if (ch < nch) {
#pragma unroll
              for (int gq = 0; gq < 4; ++gq) {
                const int col = 32 * ch + 8 * gq + cpair;
                float2 v = *reinterpret_cast<const float2*>(scr + col);
#pragma unroll
                for (int w4 = 1; w4 < 4; ++w4) {
                  const float2 o = *reinterpret_cast<const float2*>(scr + w4 * 128 + col);
                  v.x = fmaxf(v.x, o.x);
                  v.y = fmaxf(v.y, o.y);
                }
                // increase of the reference (the first tile sets it: its scores were taken against 0)
                cm[JC(ch, gq, 0)] = first ? v.x : fmaxf(v.x, 0.f);
                cm[JC(ch, gq, 1)] = first ? v.y : fmaxf(v.y, 0.f);
              }
            }
          }
          // new reference: -m -= increase (quarter 0's lanes 0-3 hold every column between them;
          // the barrier below publishes it before any thread reads nm_s again)
#pragma unroll
          for (int ch = 0; ch < 4; ++ch)
            if (ch < nch)
#pragma unroll
              for (int gq = 0; gq < 4; ++gq) {
                float* q2 = nm_s + 32 * ch + 8 * gq + cpair;
                const float2 o = first ? make_float2(0.f, 0.f) : *reinterpret_cast<const float2*>(q2);
                st_shared_f32x2_if(quarter == 0 && lane < 4, q2, o.x - cm[JC(ch, gq, 0)], o.y - cm[JC(ch, gq, 1)]);
              }
          if (!first) {
            addf = 0u;
#pragma unroll
            for (int i = 0; i < 32; ++i) {
              if ((i >> 3) < nch) {
                const bool jump = cm[i] >= 100.f;
                const float alpha = ex2_approx(-cm[i]);
                l[i] = jump ? 0.f : l[i] * alpha;
                addf |= static_cast<uint32_t>(jump) << i;
                cm[i] = alpha;
              }
            }
          }
          if (!first) {
            // O^T columns scale by alpha; the slot's previous PV completed before this S^T
            // tile was committed
#pragma unroll
            for (int ch = 0; ch < 4; ++ch) {
              if (ch < nch) {
                uint32_t o[32];
                tmem_ld_16x256b_pair(tO0 + ch * 32, tO1 + ch * 32, o);
#pragma unroll
                for (int kb = 0; kb < 4; ++kb)
#pragma unroll
                  for (int gq = 0; gq < 4; ++gq)
#pragma unroll
                    for (int c = 0; c < 2; ++c)
                      o[CI(kb, gq, c)] = __float_as_uint(__uint_as_float(o[CI(kb, gq, c)]) * cm[JC(ch, gq, c)]);
                tmem_st_16x256b_pair(tO0 + ch * 32, tO1 + ch * 32, o);
              }
            }
          }
          // every thread has read the scratch before P^T is written over it
          named_barrier_sync(bar_id, 128);
          exp_pass(true, addf);
        }
        // P^T (generic-proxy stores) becomes visible to the tensor core's operand reads
        fence_proxy_async_smem();
        tc_fence_before_sync();
        warp_arrive(&bars[KT_P_FULL + x]);
        ++sj;
      }
      // ---------------------------------------------------------- epilogue
      if (jobs > 0 && ok) ok = warp_wait(&bars[KT_O_DONE + x], (sj - 1) & 1, p.wait_ns);
      tc_fence_after_sync();
      // column sums over the warp's keys: lanes with the same lane % 4 hold the same columns
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        if ((i >> 3) < nch) {
          float v = l[i];
          v += __shfl_xor_sync(0xffffffffu, v, 4);
          v += __shfl_xor_sync(0xffffffffu, v, 8);
          v += __shfl_xor_sync(0xffffffffu, v, 16);
          l[i] = v;
        }
      }
      const int r = quarter * 32 + lane;  // this thread's column (coefficients) and O^T lane (head dim)
      if (qs) {
        // each slot finishes its own queries; scratch in its own P^T buffer (its PVs are done)
        float* sl = reinterpret_cast<float*>(pt);  // [4][128] column sums per warp
        float* coef = sl + 512;
        long long* roff = reinterpret_cast<long long*>(sl + 640);
#pragma unroll
        for (int ch = 0; ch < 4; ++ch)
          if (ch < nch)
#pragma unroll
            for (int gq = 0; gq < 4; ++gq)
              st_shared_f32x2_if(lane < 4, sl + quarter * 128 + 32 * ch + 8 * gq + cpair, l[JC(ch, gq, 0)],
                                 l[JC(ch, gq, 1)]);
        named_barrier_sync(bar_id, 128);
        {
          // every lane computes (r < 128 stays inside the scratch); only valid rows store
          const float lsum = (sl[r] + sl[128 + r]) + (sl[256 + r] + sl[384 + r]);
          const int pr = x * w.nA + r;  // packed (query, head-in-group) row
          const bool valid = r < n && pr < w.rows;
          const int qi = pr / p.grp;
          const int h = w.g * p.grp + (pr - qi * p.grp);
          const int64_t orow = (w.gm.new_row + qi) * p.h_q + h;
          if (p.lse) st_global_f32_pred(p.lse + orow, (log2f(lsum) - nm_s[r]) * kLn2, valid);
          coef[r] = 1.f / lsum;
          roff[r] = valid ? orow * D : -1;
        }
        named_barrier_sync(bar_id, 128);
        for (int c0 = 0; c0 < n; c0 += 16) {
          uint32_t o[16];
          tmem_ld_x16(tOA + x * 128 + c0, o);
#pragma unroll
          for (int c = 0; c < 16; ++c) {
            const long long ro = roff[c0 + c];
            st_global_bf16_if(ro >= 0, p.out + ro + r, __float2bfloat16_rn(__uint_as_float(o[c]) * coef[c0 + c]));
          }
        }
        tc_fence_before_sync();
        warp_arrive(&bars[KT_O_FREE + x]);
        named_barrier_sync(bar_id, 128);  // the scratch is read before the next unit writes P^T
      } else {
        // keys split: both slots hold partial states of the same queries; scratch in
        // slot B's P^T buffer once both slots' PV GEMMs are done
        named_barrier_sync(3, 256);
        float* sl = reinterpret_cast<float*>(smem + L::R + kt_pt(false, 1));  // [2][4][128]
        float* ca = sl + 1024;
        float* cb = sl + 1152;
        long long* roff = reinterpret_cast<long long*>(sl + 1280);
#pragma unroll
        for (int ch = 0; ch < 4; ++ch)
          if (ch < nch)
#pragma unroll
            for (int gq = 0; gq < 4; ++gq)
              st_shared_f32x2_if(lane < 4, sl + x * 512 + quarter * 128 + 32 * ch + 8 * gq + cpair, l[JC(ch, gq, 0)],
                                 l[JC(ch, gq, 1)]);
        named_barrier_sync(3, 256);
        const bool has_b = w.nt >= 2;  // slot B processed at least one key tile
        if (x == 0) {
          // every lane computes (r < 128 stays inside the scratch); only valid rows store
          const float la = (sl[r] + sl[128 + r]) + (sl[256 + r] + sl[384 + r]);
          const float lb = has_b ? (sl[512 + r] + sl[640 + r]) + (sl[768 + r] + sl[896 + r]) : 0.f;
          const float ma = -m_all[r], mb = -m_all[128 + r];
          const float m = lb > 0.f ? fmaxf(ma, mb) : ma;
          const float ea = ex2_approx(ma - m), eb = ex2_approx(mb - m);
          const float a = ea;
          const float b = lb > 0.f ? eb : 0.f;
          const float lsum = a * la + b * lb;
          const bool valid = r < n && r < w.rows;
          const int qi = r / p.grp;
          const int h = w.g * p.grp + (r - qi * p.grp);
          const int64_t orow = (w.gm.new_row + qi) * p.h_q + h;
          if (p.lse) st_global_f32_pred(p.lse + orow, (m + log2f(lsum)) * kLn2, valid);
          ca[r] = a / lsum;
          cb[r] = b / lsum;
          roff[r] = valid ? orow * D : -1;
        }
        named_barrier_sync(3, 256);
        // slot x writes columns [x n / 2, (x + 1) n / 2)
        const int hn = n >> 1;
        for (int c0 = x * hn; c0 < (x + 1) * hn; c0 += 8) {
          uint32_t oa[8], ob[8];
          tmem_ld_x8(tOA + c0, oa);
          if (has_b) tmem_ld_x8(tOB + c0, ob);
#pragma unroll
          for (int c = 0; c < 8; ++c) {
            const long long ro = roff[c0 + c];
            float v = __uint_as_float(oa[c]) * ca[c0 + c];
            if (has_b) v = fmaf(__uint_as_float(ob[c]), cb[c0 + c], v);
            st_global_bf16_if(ro >= 0, p.out + ro + r, __float2bfloat16_rn(v));
          }
        }
        tc_fence_before_sync();
        named_barrier_sync(3, 256);  // both slots have read both accumulators and the scratch
        warp_arrive(&bars[KT_O_FREE + x]);
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

}  // namespace

ssm_status launch_attn_keytile(const AttnMaps& m, const AttnParams& p, int grid, cudaStream_t st) {
  // the warpgroup register split assumes the compiled register count
  static std::atomic<int> regs_ok{0};  // 0 unknown, 1 ok, 2 mismatch
  int st_regs = regs_ok.load();
  if (st_regs == 0) {
    cudaFuncAttributes fa;
    if (cudaFuncGetAttributes(&fa, attn_keytile_kernel) != cudaSuccess) return SSM_ERR_CUDA;
    st_regs = fa.numRegs == kLaunchRegs ? 1 : 2;
    regs_ok.store(st_regs);
  }
  if (st_regs != 1) return SSM_ERR_UNSUPPORTED;
  static std::atomic<uint64_t> attr_set{0};
  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return SSM_ERR_CUDA;
  const uint64_t bit = 1ull << (dev & 63);
  if (!(attr_set.load() & bit)) {
    if (cudaFuncSetAttribute(attn_keytile_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, KtLayout::ALLOC) !=
        cudaSuccess)
      return SSM_ERR_CUDA;
    attr_set.fetch_or(bit);
  }
  attn_keytile_kernel<<<grid, kAttnThreads, KtLayout::ALLOC, st>>>(m.q128, m.q96, m.kc, m.vc, m.kn, m.vn, m.kc128,
                                                                    m.vc128, m.kn128, m.vn128, p);
  return launch_status();
}

}  // namespace ssm
