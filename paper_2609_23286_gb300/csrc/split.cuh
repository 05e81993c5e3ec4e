// The attention's stream-K split and the merge of units cut between CTAs.
//
// The (unit, key tile) sequence -- a unit is a pair of 128-row query tiles
// (unit_tiles), run over every key tile of [bank ; frame] -- runs in one or
// two phases, each cut into G contiguous ranges of about equal cost
// (attn_split_bounds), CTA b taking [x[p][b], x[p][b + 1]) in phase p.  A
// unit cut by a CTA boundary leaves, from each CTA that holds part of it, one
// normalised partial per query row, (O_p, LSE_p), in the CTA's slot 2p (the
// unit is the CTA's first piece of phase p) or 2p + 1 (its last piece), O_p in
// bf16 and LSE_p in fp32.  The merge of Eq. 3
// over the pieces is the log-sum-exp combination
//     LSE = log sum_p exp(LSE_p),   O = sum_p exp(LSE_p - LSE) O_p,
// folded in CTA order, so the result does not depend on which CTA finished
// first.  The attention kernel writes the partials; attn_combine_kernel,
// launched right behind it, merges them.

#pragma once

#include <cuda_bf16.h>

#include "kernels.h"
#include "ptx.cuh"

namespace regmem_dev {
namespace split {

constexpr int kRows = kTile;            // rows of a query tile
constexpr int kUnitRowsS = kUnitRows;   // rows of a unit (two tiles)
constexpr int kMergeThreads = 4;        // threads per row in a merge (16 channels each)
constexpr int kPrefetch = 2;            // pieces whose loads are issued together

using Layout = SplitLayout;

// Phase of tile x.
__host__ __device__ __forceinline__ int phase_of(const SplitBounds& sb, long long x) {
  return sb.P > 1 && x >= sb.pbeg[1] ? 1 : 0;
}

// CTA whose range of phase p contains tile x (binary search of the cuts).
__host__ __device__ __forceinline__ int cta_of(const SplitBounds& sb, int p, int G, long long x) {
  int lo = 0, hi = G - 1;  // sb.x[p][lo] <= x < sb.x[p][hi + 1]
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (sb.x[p][mid] <= x) lo = mid;
    else hi = mid - 1;
  }
  return lo;
}

// The CTAs holding a split unit of phase p: b_lo .. b_hi, and the slot of
// b_lo's piece (every later CTA holds the unit as its first piece of the
// phase, slot 2p).
struct Pieces {
  int b_lo, b_hi, which_lo, p, slots;
};

// Row `r` (0..255 within the unit) of piece i (0-based from b_lo) in the
// partial arrays.
__device__ __forceinline__ size_t piece_row(const Pieces& pc, int i, int r) {
  const int bb = pc.b_lo + i;
  const int which = i == 0 ? pc.which_lo : 0;
  return ((size_t)bb * pc.slots + 2 * pc.p + which) * kUnitRowsS + r;
}

// Merges 16 channels (quarter qtr) of row r of tile t of split unit u and
// writes them to out (bf16); the thread with qtr == 0 also writes the LSE.
// The bf16 partials add one rounding (relative 2^-9) to the rows of split
// units before the fp32 fold.
__device__ __forceinline__ void merge_row(const Layout& s, const Pieces& pc, int u, int t, int r,
                                          int qtr) {
  const UnitTiles ut = unit_tiles(u, s.nqt, s.H);
  const int h = t ? ut.h1 : ut.h0;
  const int q = (t ? ut.qt1 : ut.qt0) * kRows + r;
  const int ur = t * kRows + r;  // row within the unit
  const int np = pc.b_hi - pc.b_lo + 1;
  if (!dev_check(pc.b_lo >= 0 && pc.b_hi < s.G && np >= 2 && 2 * pc.p + 1 < pc.slots, s.status)) return;
  // the partials were kept in L2 for this read; afterwards they may go
  const uint64_t pol = ptx::l2_policy_evict_first();
  float lp[kPrefetch];
  uint4 v[kPrefetch][2];
#pragma unroll
  for (int i = 0; i < kPrefetch; ++i) {
    if (i < np) {
      const size_t pr = piece_row(pc, i, ur);
      lp[i] = ptx::ld_global_hint(s.part_lse + pr, pol);
      const uint4* src = reinterpret_cast<const uint4*>(s.part_o + pr * kHeadDim) + qtr * 2;
#pragma unroll
      for (int c = 0; c < 2; ++c) v[i][c] = __ldcg(src + c);
    }
  }
  float m = -INFINITY;
#pragma unroll
  for (int i = 0; i < kPrefetch; ++i)
    if (i < np) m = fmaxf(m, lp[i]);
  for (int i = kPrefetch; i < np; ++i) m = fmaxf(m, ptx::ld_global_hint(s.part_lse + piece_row(pc, i, ur), pol));
  float den = 0.f, acc[16];
#pragma unroll
  for (int c = 0; c < 16; ++c) acc[c] = 0.f;
  auto fold = [&](float l, const uint4 (&w)[2]) {
    const float a = ptx::ex2((l - m) * 1.4426950408889634f);
    den += a;
#pragma unroll
    for (int c = 0; c < 2; ++c) {
      const uint32_t ww[4] = {w[c].x, w[c].y, w[c].z, w[c].w};
#pragma unroll
      for (int e = 0; e < 4; ++e) {
        acc[c * 8 + e * 2 + 0] += __uint_as_float(ww[e] << 16) * a;
        acc[c * 8 + e * 2 + 1] += __uint_as_float(ww[e] & 0xFFFF0000u) * a;
      }
    }
  };
#pragma unroll
  for (int i = 0; i < kPrefetch; ++i)
    if (i < np) fold(lp[i], v[i]);
  for (int i = kPrefetch; i < np; ++i) {  // units cut into more pieces than are prefetched
    const size_t pr = piece_row(pc, i, ur);
    const uint4* src = reinterpret_cast<const uint4*>(s.part_o + pr * kHeadDim) + qtr * 2;
    uint4 w[2];
#pragma unroll
    for (int c = 0; c < 2; ++c) w[c] = __ldcg(src + c);
    fold(ptx::ld_global_hint(s.part_lse + pr, pol), w);
  }
  if (q >= s.N) return;
  const float inv = 1.f / den;
  uint4* o = reinterpret_cast<uint4*>(s.out + ((size_t)q * s.H + h) * kHeadDim) + qtr * 2;
#pragma unroll
  for (int c8 = 0; c8 < 2; ++c8) {
    uint4 w4;
    w4.x = ptx::pack_bf16x2(acc[c8 * 8 + 0] * inv, acc[c8 * 8 + 1] * inv);
    w4.y = ptx::pack_bf16x2(acc[c8 * 8 + 2] * inv, acc[c8 * 8 + 3] * inv);
    w4.z = ptx::pack_bf16x2(acc[c8 * 8 + 4] * inv, acc[c8 * 8 + 5] * inv);
    w4.w = ptx::pack_bf16x2(acc[c8 * 8 + 6] * inv, acc[c8 * 8 + 7] * inv);
    o[c8] = w4;
  }
  if (qtr == 0) s.lse[(size_t)h * s.N + q] = m + __logf(den);
}

// Merge job j (0 .. 2 P (G - 1) - 1) of phase p = j / (2 (G - 1)), with
// jj = j mod 2 (G - 1): query tile jj & 1 of the unit cut by the phase's
// boundary between CTAs jj / 2 and jj / 2 + 1, unless that boundary is not
// strictly inside a unit or an earlier boundary cuts the same unit.
// prepare_job needs only the layout (it can run before the attention's
// partials are complete); run_job merges every row of the tile with a group
// of NT threads (thread index tid).
struct Job {
  int u, t;  // u < 0: nothing to merge
  Pieces pc;
};
// Whether job j merges anything (host and device).
__host__ __device__ inline int job_count(const Layout& s) { return 2 * s.bnd.P * (s.G - 1); }
__host__ __device__ inline bool job_live(const Layout& s, int j) {
  const int p = j / (2 * (s.G - 1)), jj = j - p * 2 * (s.G - 1);
  const int bnd = jj / 2 + 1;
  const long long xb = s.bnd.x[p][bnd];
  const long long u = xb / s.nkv;
  const long long x0 = u * s.nkv;
  if (xb == x0 || s.bnd.x[p][bnd - 1] > x0) return false;
  return (jj & 1) == 0 || unit_tiles(u, s.nqt, s.H).has1;
}
__device__ __forceinline__ Job prepare_job(const Layout& s, int j) {
  Job jb;
  jb.u = -1;
  jb.t = j & 1;
  if (j < 0 || j >= job_count(s) || !job_live(s, j)) return jb;
  const int p = j / (2 * (s.G - 1)), jj = j - p * 2 * (s.G - 1);
  const int bnd = jj / 2 + 1;
  const long long x0 = s.bnd.x[p][bnd] / s.nkv * s.nkv;
  jb.u = (int)(x0 / s.nkv);
  jb.pc.p = p;
  jb.pc.slots = s.bnd.slots;
  jb.pc.b_lo = bnd - 1;  // the CTA holding the unit's first tile
  jb.pc.b_hi = cta_of(s.bnd, p, s.G, x0 + s.nkv - 1);
  jb.pc.which_lo = s.bnd.x[p][jb.pc.b_lo] == x0 ? 0 : 1;
  return jb;
}
template <int NT>
__device__ __forceinline__ void run_job(const Layout& s, const Job& jb, int tid) {
  static_assert(NT % kMergeThreads == 0, "whole rows per pass");
  if (jb.u < 0) return;
  constexpr int RPP = NT / kMergeThreads;  // rows per pass
  for (int r = tid / kMergeThreads; r < kRows; r += RPP)
    merge_row(s, jb.pc, jb.u, jb.t, r, tid % kMergeThreads);
}

}  // namespace split
}  // namespace regmem_dev
