// Per-head admission into the regulated memory (Eq. 6 with the head-specific
// retention of Sec. 3.3): among the candidate tokens, the k with the largest
// saliency -- order (saliency descending, token index ascending), so ties go
// to the lower index -- appended to the head's bank in ascending token order.
// Saliency values map to order-preserving 32-bit keys.  Two exact selections:
//
// * distributed (k <= 32, the regime of a ~1% budget): every block holding a
//   128-key tile of a head sorts its candidates, packed as (key << 32 |
//   ~token) so the order is a plain descending order of distinct 64-bit
//   values, with warp bitonic sorts and merges, and stores its best 32; the
//   last block of the head merges the tiles' lists.  Each step is a few
//   shuffle stages with eight-way independent work, which suits a GPU whose
//   single-block selections are bound by dependent-instruction latency.
// * radix (any k, one block per head): the k-th largest key T is built four
//   bits at a time from the top (eight steps; in each, every thread counts its
//   keys that share T's chosen digits and have the next digit >= v for
//   v = 1..15, warp butterflies sum the counts, and one warp picks the largest
//   digit that still leaves >= k keys at or above T).  Every key above T is
//   admitted; of the keys equal to T the lowest token indices fill the
//   remaining slots (a block scan in token order), and a second scan over the
//   admitted flags gives each admitted token its slot.  Thread t owns the
//   contiguous key slice [t * per, t * per + per), so the scans follow token
//   order.
#pragma once

#include "kernels.h"

namespace regmem_dev {
namespace sel {

// float -> unsigned key with the same order (negative values reversed).
__device__ __forceinline__ uint32_t order_bits(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive prefix sum over the block of one value per thread; `ws` holds
// THREADS / 32 ints.
template <int THREADS>
__device__ __forceinline__ int block_exclusive_scan(int v, int* ws) {
  constexpr int WARPS = THREADS / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) ws[warp] = x;
  __syncthreads();
  int base = 0;
#pragma unroll
  for (int w = 0; w < WARPS; ++w) base += (w < warp) ? ws[w] : 0;
  __syncthreads();  // ws may be reused by the next scan
  return base + x - v;
}

// Sums each of 16 per-lane values over the warp with 16 shuffles (instead of
// 16 reductions of 5 shuffles each).  Returns, on lane l, the warp sum of
// value (l >> 1): at level j the lanes with bit (4 - j) of the lane set keep
// the upper half of the remaining values, the others the lower half.
__device__ __forceinline__ int warp_sum16(const int (&s)[16], int lane) {
  int a[8], b[4], c[2];
  {
    const bool up = lane & 16;
#pragma unroll
    for (int j = 0; j < 8; ++j) {
      const int send = up ? s[j] : s[j + 8];
      const int keep = up ? s[j + 8] : s[j];
      a[j] = keep + __shfl_xor_sync(0xffffffffu, send, 16);
    }
  }
  {
    const bool up = lane & 8;
#pragma unroll
    for (int j = 0; j < 4; ++j) {
      const int send = up ? a[j] : a[j + 4];
      const int keep = up ? a[j + 4] : a[j];
      b[j] = keep + __shfl_xor_sync(0xffffffffu, send, 8);
    }
  }
  {
    const bool up = lane & 4;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int send = up ? b[j] : b[j + 2];
      const int keep = up ? b[j + 2] : b[j];
      c[j] = keep + __shfl_xor_sync(0xffffffffu, send, 4);
    }
  }
  const bool up = lane & 2;
  int d = (up ? c[1] : c[0]) + __shfl_xor_sync(0xffffffffu, up ? c[0] : c[1], 2);
  d += __shfl_xor_sync(0xffffffffu, d, 1);
  return d;  // value index: bit 3 = lane bit 4, bit 2 = lane bit 3, bit 1 = lane bit 2, bit 0 = lane bit 1
}

// Shared words the radix selection needs in `red` for a block of THREADS.
template <int THREADS>
constexpr int red_words() { return 2 * 16 * THREADS / 32; }

// keys[0..n) in shared memory, 1 <= k <= n.  Writes the positions (0..n-1)
// of the k admitted keys, ascending, to ord[0..k) (shared memory) and ends
// with a barrier.  Shared scratch: `red` 2 * 16 * THREADS / 32 ints, `ws`
// THREADS / 32 ints, `bc` 2 ints.
template <int THREADS>
__device__ __forceinline__ void select_topk_radix(const uint32_t* keys, int n, int k, int* ord, int* red, int* ws, int* bc) {
  constexpr int WARPS = THREADS / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int per = (n + THREADS - 1) / THREADS;
  const int first = threadIdx.x * per;
  const int cnt = max(0, min(per, n - first));
  uint32_t T = 0;  // digits of the k-th largest key chosen so far (lower bits zero)
  int above = 0;   // keys whose chosen digits already exceed T's: all admitted
#pragma unroll 1
  for (int shift = 28; shift >= 0; shift -= 4) {
    const uint32_t hmask = shift == 28 ? 0u : ~0u << (shift + 4);
    int s[16];  // s[v]: my keys with T's high digits and next digit >= v (v >= 1)
#pragma unroll
    for (int v = 0; v < 16; ++v) s[v] = 0;
#pragma unroll 4
    for (int i = 0; i < cnt; ++i) {
      const uint32_t key = keys[first + i];
      const bool m = ((key ^ T) & hmask) == 0;
      const uint32_t d = (key >> shift) & 15u;
#pragma unroll
      for (int v = 1; v < 16; ++v) s[v] += (m && d >= (uint32_t)v) ? 1 : 0;
    }
    int* r = red + ((shift >> 2) & 1) * (16 * WARPS);
    // warp sums of the 16 counts in four butterfly halvings plus one step: at
    // each level a lane keeps one half of its values, receives the partner's
    // copy of that half and adds; lane l ends with the sum of value v(l)
    {
      const int vl = warp_sum16(s, lane);
      if ((lane & 1) == 0) r[warp * 16 + (lane >> 1)] = vl;
    }
    __syncthreads();
    if (warp == 0) {
      int tot = 0;  // lane v: block count for digit >= v (non-increasing in v)
      if (lane >= 1 && lane < 16)
        for (int w = 0; w < WARPS; ++w) tot += r[w * 16 + lane];
      const bool q = lane == 0 || (lane < 16 && above + tot >= k);  // v = 0 always qualifies
      const int vstar = 31 - __clz(__ballot_sync(0xffffffffu, q));
      const int more = __shfl_sync(0xffffffffu, tot, vstar + 1);  // digit > vstar (0 past 15)
      if (lane == 0) {
        bc[0] = vstar;
        bc[1] = above + more;
      }
    }
    __syncthreads();
    T |= (uint32_t)bc[0] << shift;
    above = bc[1];
  }
  // T is the k-th largest key; `above` keys are strictly greater
  int n_eq = 0;
  for (int i = 0; i < cnt; ++i) n_eq += keys[first + i] == T;
  const int krem = k - above;  // keys equal to T to admit, >= 1
  const int eq_rank = block_exclusive_scan<THREADS>(n_eq, ws);
  int n_sel = 0;
  {
    int er = eq_rank;
    for (int i = 0; i < cnt; ++i) {
      const uint32_t key = keys[first + i];
      n_sel += (key > T) || (key == T && er++ < krem);
    }
  }
  int slot = block_exclusive_scan<THREADS>(n_sel, ws);
  {
    int er = eq_rank;
    for (int i = 0; i < cnt; ++i) {
      const uint32_t key = keys[first + i];
      if ((key > T) || (key == T && er++ < krem)) ord[slot++] = first + i;
    }
  }
  __syncthreads();
}

// ---------------------------------------------------------------------------
// Distributed selection for k <= kListK (the admission budget is about 1% of
// the frame): every block that holds a 128-key tile of a head sorts its
// candidates and keeps its top kListK; the last block of the head merges the
// tiles' lists.  A candidate is the 64-bit value (key << 32) | ~token, so the
// order (saliency descending, token ascending) is a plain descending order
// of distinct values; 0 marks "no candidate" (every real key is >= 2^31).
// The union of the per-tile top-k holds the head's top-k.
constexpr int kListK = kFusedMaxK;

__device__ __forceinline__ uint64_t pack_candidate(float s, int token) {
  return ((uint64_t)order_bits(s) << 32) | (uint32_t)~(uint32_t)token;
}
__device__ __forceinline__ int candidate_token(uint64_t v) { return (int)~(uint32_t)v; }

// Bitonic sort of one value per lane, descending across lanes 0..31.
__device__ __forceinline__ uint64_t warp_sort_desc(uint64_t v, int lane) {
#pragma unroll
  for (int size = 2; size <= 32; size <<= 1) {
    const bool desc = (lane & size) == 0;  // direction of this lane's block (all descending at 32)
#pragma unroll
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      const uint64_t o = __shfl_xor_sync(0xffffffffu, v, stride);
      const bool lower = (lane & stride) == 0;
      v = (lower == desc) ? (v > o ? v : o) : (v < o ? v : o);
    }
  }
  return v;
}

// Top 32 of two descending lane-sorted lists, descending: the elementwise
// maximum of a and reversed b is bitonic and holds the top 32; five merge
// stages sort it.
__device__ __forceinline__ uint64_t warp_merge_top(uint64_t a, uint64_t b, int lane) {
  const uint64_t br = __shfl_sync(0xffffffffu, b, 31 - lane);
  uint64_t v = a > br ? a : br;
#pragma unroll
  for (int stride = 16; stride > 0; stride >>= 1) {
    const uint64_t o = __shfl_xor_sync(0xffffffffu, v, stride);
    v = ((lane & stride) == 0) ? (v > o ? v : o) : (v < o ? v : o);
  }
  return v;
}

// Block of THREADS (one candidate value per thread): writes the block's top
// kListK values, descending, to out[0..kListK).  `lists`: shared scratch of
// THREADS uint64.  Ends with a barrier.
template <int THREADS>
__device__ __forceinline__ void block_top_list(uint64_t v, uint64_t* lists, uint64_t* out) {
  constexpr int WARPS = THREADS / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  lists[warp * 32 + lane] = warp_sort_desc(v, lane);
  __syncthreads();
  if (warp == 0) {
    uint64_t t = lists[lane];
#pragma unroll
    for (int w = 1; w < WARPS; ++w) t = warp_merge_top(t, lists[w * 32 + lane], lane);
    out[lane] = t;
  }
  __syncthreads();
}

// Last block of a head: merges the ntiles lists of kListK values (global,
// written by other blocks of the grid) and writes the k admitted positions
// relative to cand_lo, ascending, to ord[0..k).  `lists`: shared scratch of
// THREADS uint64.  Ends with a barrier.
template <int THREADS>
__device__ __forceinline__ void merge_head_lists(const uint64_t* head_lists, int ntiles, int k,
                                                 int cand_lo, uint64_t* lists, int* ord) {
  constexpr int WARPS = THREADS / 32;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  uint64_t t = 0;
  for (int i = warp; i < ntiles; i += WARPS)
    t = warp_merge_top(t, __ldcg(reinterpret_cast<const unsigned long long*>(head_lists) + i * kListK + lane), lane);
  lists[warp * 32 + lane] = t;
  __syncthreads();
  if (warp == 0) {
    t = lists[lane];
#pragma unroll
    for (int w = 1; w < WARPS; ++w) t = warp_merge_top(t, lists[w * 32 + lane], lane);
    // lanes 0..k-1 hold the admitted candidates; sort their tokens ascending
    uint64_t pos = lane < k ? (uint64_t)candidate_token(t) : ~0ull;
    // ascending bitonic sort: the descending sort of the complement
    pos = ~warp_sort_desc(~pos, lane);
    if (lane < k) ord[lane] = (int)pos - cand_lo;
  }
  __syncthreads();
}

// Dispatch for the single-block selection over keys in shared memory.
// `red` must hold red_words<THREADS>() words.
template <int THREADS>
__device__ __forceinline__ void select_topk(const uint32_t* keys, int n, int k, int* ord, int* red,
                                            int* ws, int* bc) {
  select_topk_radix<THREADS>(keys, n, k, ord, red, ws, bc);
}

// Loads the candidates' saliency of head h into keys[0..n) (L2 reads: the
// values may have been written by other blocks of the same grid).
template <int THREADS>
__device__ __forceinline__ void load_keys(const float* sal_h, int n, uint32_t* keys) {
#pragma unroll 4
  for (int i = threadIdx.x; i < n; i += THREADS) keys[i] = order_bits(__ldcg(sal_h + i));
  __syncthreads();
}

// Appends the admitted rows (token = cand_lo + ord[r]) of head h after the M
// rows already in its bank, K then V, 16 bytes per thread and step; writes
// the token indices to idx_out[h][k] when given.
template <int THREADS>
__device__ __forceinline__ void append_rows(const AdmitArgs& a, int h, const int* ord) {
  constexpr int HD = kHeadDim;
  if (a.idx_out)
    for (int r = threadIdx.x; r < a.k; r += THREADS) a.idx_out[(size_t)h * a.k + r] = a.cand_lo + ord[r];
  const int work = a.k * 8 * 2;
  for (int w = threadIdx.x; w < work; w += THREADS) {
    const int which = w / (a.k * 8);
    const int rem = w - which * a.k * 8;
    const int r = rem >> 3, c = rem & 7;
    const int tok = a.cand_lo + ord[r];
    if (!dev_check(tok >= a.cand_lo && tok < a.N && a.M + r < a.cap, a.status)) continue;
    const __nv_bfloat16* src = (which ? a.V : a.K) + ((size_t)tok * a.H + h) * HD;
    __nv_bfloat16* dst = (which ? a.bankV : a.bankK) + ((size_t)h * a.cap + a.M + r) * HD;
    reinterpret_cast<uint4*>(dst)[c] = reinterpret_cast<const uint4*>(src)[c];
  }
}

}  // namespace sel
}  // namespace regmem_dev
