// Regulated causal attention with row log-sum-exp on the 5th-generation tensor
// cores (Eq. 2 / Eq. 3, LSE of Sec. 3.3 "FlashAttention-Compatible Saliency
// Estimation").
//
// For every head h and 128-row query tile the kernel computes
//     O = softmax(Q K_c^T * scale) V_c,  LSE_i = log sum_j exp(Z_ij)
// over K_c = [bank rows of head h (M of them) ; the frame's N keys], with no
// mask inside the frame (frame-granular causality).  The key sequence is cut
// into 128-row tiles: ceil(M/128) bank tiles followed by ceil(N/128) frame
// tiles, each possibly ragged (columns past the valid count are masked).
//
// Work split (stream-K over the key dimension): the (unit, key tile) space,
// unit = (head, query tile), is cut into `grid` contiguous equal ranges, one
// per CTA.  A unit whose key tiles all fall in one CTA is finished there (O in
// bf16 and LSE written directly); a unit cut between CTAs leaves normalised
// fp32 partials (O_p, LSE_p) that attn_combine_kernel merges.
//
// CTA layout (256 threads = 8 warps, 2 CTAs per SM, so each SM sub-partition
// runs four softmax warps): every query row of the 128-row tile is shared by
// two threads, one per half of the 128 key columns -- warp w owns TMEM lanes
// 32*(w%4)..+31 and columns 64*(w/4)..+63 of S (and 32*(w/4)..+31 of O).
// The two threads of a row exchange their partial row max through shared
// memory behind a 64-thread named barrier; each keeps a partial row sum that
// is combined once, in the epilogue.  Thread 0 also issues the TMA loads
// (K through a 3-stage ring, V through a 2-stage ring) and the tcgen05 MMAs.
// TMEM (256 columns): S = Q K^T fp32 [0,128), P bf16 packed [128,192),
// O fp32 [192,256).  Q K^T is an SS-MMA (both operands K-major in smem);
// P V is a TS-MMA (P from TMEM, V MN-major in smem).
// Pipelining inside a CTA: as soon as every thread has pulled its half of
// S(t) into registers, Q K^T of tile t+1 is issued, so the tensor core
// computes S(t+1) while the softmax of tile t runs; P V(t) is issued once P(t)
// is in TMEM.  Two mbarriers pace this: s_bar completes per Q K^T, o_bar per
// P V.  P(t) is stored only after P V(t-1) has finished reading the P
// columns; at that point V(t-1)'s stage is refilled with V(t+1) and K(t-1)'s
// stage with K(t+2).
// The softmax keeps a stale running max and only rescales O when the max
// grows by more than 2^8, so exp values stay <= 256.

#include "kernels.h"
#include "ptx.cuh"

namespace regmem_dev {
using namespace ptx;

namespace {

constexpr int BM = kTile, BN = kTile, HD = kHeadDim;
constexpr int KSTAGES = 3, VSTAGES = 2;
constexpr int TILE_BYTES = BM * HD * 2;  // 16 KB bf16 tile
constexpr int THREADS = 256;
constexpr uint32_t TMEM_COLS = 256, TM_S = 0, TM_P = 128, TM_O = 192;
constexpr uint64_t WAIT_NS = 2000000000ull;   // 2 s: a hung pipeline gives up
constexpr uint64_t DRAIN_NS = 200000000ull;   // 0.2 s for draining on abort
constexpr float RESCALE_LOG2 = 8.0f;
constexpr uint32_t IDESC_QK = idesc_bf16_f32(128, 128, false, false);
constexpr uint32_t IDESC_PV = idesc_bf16_f32(128, 64, false, true);

struct Smem {
  uint8_t q[TILE_BYTES];
  uint8_t k[KSTAGES][TILE_BYTES];
  uint8_t v[VSTAGES][TILE_BYTES];
  float xch[2][BM];  // per-row partial max / partial sum of each column half
  uint64_t q_full, k_full[KSTAGES], v_full[VSTAGES], s_bar, o_bar, fin_bar;
  uint32_t tmem_base;
  int abort_flag;
  int never;  // always 0: abort word for waits that must not be cut short
};
// Tiles + exchange + barriers, rounded to 128 B; the dynamic shared window is
// requested 1 KB aligned (128-byte swizzle atoms need it) and checked at run
// time.  About 97 KB, so two CTAs share an SM.
constexpr size_t SMEM_BYTES = (sizeof(Smem) + 127) & ~size_t(127);

struct Params {
  int N, H, M;
  int nb, nkv, nqt;
  long long total;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  float* part_o;
  float* part_lse;
  int* status;
};

__device__ __forceinline__ long long range_begin(int b, int G, long long T) {
  return (long long)b * T / G;
}

__device__ __forceinline__ int tile_valid(const Params& p, int j) {
  return j < p.nb ? min(BN, p.M - j * BN) : min(BN, p.N - (j - p.nb) * BN);
}

__device__ __forceinline__ void issue_qk(uint32_t d, uint32_t sq, uint32_t sk) {
#pragma unroll
  for (int kk = 0; kk < HD / 16; ++kk)
    mma_ss(d, sdesc_sw128(sq + kk * 32), sdesc_sw128(sk + kk * 32), IDESC_QK, kk > 0);
}

// Key tile x (global linear index over (unit, key tile)) -> head and source.
struct TileSrc {
  const CUtensorMap* map;
  int c1, c2;
};
__device__ __forceinline__ TileSrc tile_src(const Params& p, long long x, const CUtensorMap* fr,
                                           const CUtensorMap* bank) {
  const int u = (int)(x / p.nkv);
  const int j = (int)(x - (long long)u * p.nkv);
  const int h = u / p.nqt;
  if (j < p.nb) return {bank, j * BN, h};         // bank rows: (channel, row, head)
  return {fr, h, (j - p.nb) * BN};                // frame rows: (channel, head, token)
}

__device__ __forceinline__ void load_k(Smem& sm, const Params& p, const CUtensorMap* tmK,
                                       const CUtensorMap* tmBK, long long x, int st) {
  const TileSrc t = tile_src(p, x, tmK, tmBK);
  const uint32_t bar = smem_addr(&sm.k_full[st]);
  mbar_arrive_expect_tx(bar, TILE_BYTES);
  tma_load_3d(smem_addr(sm.k[st]), t.map, bar, 0, t.c1, t.c2);
}

__device__ __forceinline__ void load_v(Smem& sm, const Params& p, const CUtensorMap* tmV,
                                       const CUtensorMap* tmBV, long long x, int st) {
  const TileSrc t = tile_src(p, x, tmV, tmBV);
  const uint32_t bar = smem_addr(&sm.v_full[st]);
  mbar_arrive_expect_tx(bar, TILE_BYTES);
  tma_load_3d(smem_addr(sm.v[st]), t.map, bar, 0, t.c1, t.c2);
}

__device__ __forceinline__ void load_q(Smem& sm, const Params& p, const CUtensorMap* tmQ, int u) {
  const int h = u / p.nqt, qt = u - h * p.nqt;
  mbar_arrive_expect_tx(smem_addr(&sm.q_full), TILE_BYTES);
  tma_load_3d(smem_addr(sm.q), tmQ, smem_addr(&sm.q_full), 0, h, qt * BM);
}

__global__ void __launch_bounds__(THREADS, 2)
    attn_fwd_kernel(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const __grid_constant__ CUtensorMap tmV, const __grid_constant__ CUtensorMap tmBK,
                    const __grid_constant__ CUtensorMap tmBV, const Params p) {
  extern __shared__ __align__(1024) uint8_t smem_raw[];
  if ((smem_addr(smem_raw) & 1023u) != 0) {  // uniform for the whole CTA
    if (threadIdx.x == 0) atomicOr(p.status, kStatusSmemAlign);
    return;
  }
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &sm.abort_flag;
  volatile int* never = &sm.never;
  const bool issuer = (tid == 0);

  const int G = gridDim.x, b = blockIdx.x;
  const long long x_begin = range_begin(b, G, p.total), x_end = range_begin(b + 1, G, p.total);
  const int nkv = p.nkv;
  const int u_first = (int)(x_begin / nkv);
  const uint32_t sq = smem_addr(sm.q);
  const uint32_t b_qfull = smem_addr(&sm.q_full);
  const uint32_t b_s = smem_addr(&sm.s_bar), b_o = smem_addr(&sm.o_bar);
  const uint32_t b_fin = smem_addr(&sm.fin_bar);

  // tiles whose K / V loads have been issued (issued in order 0, 1, 2, ...)
  // and Q loads issued (issuer only), for the final drain
  int nk = 0, nv = 0, q_issued = 0;
  if (issuer) {
    sm.abort_flag = 0;
    sm.never = 0;
    mbar_init(b_qfull, 1);
    for (int s = 0; s < KSTAGES; ++s) mbar_init(smem_addr(&sm.k_full[s]), 1);
    for (int s = 0; s < VSTAGES; ++s) mbar_init(smem_addr(&sm.v_full[s]), 1);
    mbar_init(b_s, 1);
    mbar_init(b_o, 1);
    mbar_init(b_fin, 1);
    fence_barrier_init();
    prefetch_tmap(&tmQ);
    prefetch_tmap(&tmK);
    prefetch_tmap(&tmV);
    prefetch_tmap(&tmBK);
    prefetch_tmap(&tmBV);
    load_q(sm, p, &tmQ, u_first);
    ++q_issued;
    for (; nk < KSTAGES - 1 && x_begin + nk < x_end; ++nk) load_k(sm, p, &tmK, &tmBK, x_begin + nk, nk);
    for (; nv < VSTAGES && x_begin + nv < x_end; ++nv) load_v(sm, p, &tmV, &tmBV, x_begin + nv, nv);
  }
  if (warp == 0) {
    tmem_alloc(smem_addr(&sm.tmem_base), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  const int quarter = warp & 3, half = warp >> 2;
  const int row = quarter * 32 + lane;  // query row inside the tile = TMEM lane
  const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
  const uint32_t s_col = TM_S + 64 * half, p_col = TM_P + 32 * half, o_col = TM_O + 32 * half;
  const int pair_bar = 1 + quarter;     // named barrier of warps quarter and quarter+4
  const float c = p.scale_log2;
  int it = 0, piece = 0;                // it: tile counter inside this CTA's range
  uint32_t s_phase = 0, o_phase = 0;
  bool stop = false;
  for (long long x = x_begin; x < x_end && !stop;) {
    const int u = (int)(x / nkv);
    const int j0 = (int)(x - (long long)u * nkv);
    const int j1 = (int)min((long long)nkv, j0 + (x_end - x));
    const int h = u / p.nqt, qt = u - h * p.nqt;
    const int n = j1 - j0;
    if (issuer) {
      bool ok = mbar_wait(b_qfull, piece & 1, abort_flag, WAIT_NS);
      const int st = it % KSTAGES;
      if (ok) ok = mbar_wait(smem_addr(&sm.k_full[st]), (it / KSTAGES) & 1, abort_flag, WAIT_NS);
      if (ok) issue_qk(tmem + TM_S, sq, smem_addr(sm.k[st]));
      mma_commit(b_s);
    }
    float m_used = -INFINITY;  // running max of the logits, scaled to log2 units
    float l = 0.f;             // this thread's half of the running row sum
    for (int jj = 0; jj < n; ++jj, ++it) {
      const int j = j0 + jj;
      const bool ok = mbar_wait(b_s, s_phase, abort_flag, WAIT_NS);  // S(it) is in TMEM
      s_phase ^= 1;
      tc_fence_after();
      uint32_t sr[64];
      if (ok) tmem_ld64(tmem + lane_off + s_col, sr);
      tc_fence_before();
      // Every thread holds its half of the S row now: the S columns are free.
      if (__syncthreads_or(!ok || *abort_flag)) {
        stop = true;
        break;
      }
      if (issuer) {
        tc_fence_after();
        if (jj + 1 < n) {
          const int st2 = (it + 1) % KSTAGES;
          if (mbar_wait(smem_addr(&sm.k_full[st2]), ((it + 1) / KSTAGES) & 1, abort_flag, WAIT_NS))
            issue_qk(tmem + TM_S, sq, smem_addr(sm.k[st2]));
          mma_commit(b_s);
        } else if (x + n < x_end) {
          // the last Q K^T of this unit has completed: bring in the next Q
          load_q(sm, p, &tmQ, u + 1);
          ++q_issued;
        }
        // Q K^T(it) has completed, so K(it-1)'s stage is free: refill it
        // with K(it+2).
        if (x_begin + nk < x_end) {  // nk == it + KSTAGES - 1 here
          load_k(sm, p, &tmK, &tmBK, x_begin + nk, nk % KSTAGES);
          ++nk;
        }
      }
      const int valid = tile_valid(p, j) - 64 * half;  // valid columns of this half
      if (valid < 64) {
#pragma unroll
        for (int i = 0; i < 64; ++i)
          if (i >= valid) sr[i] = __float_as_uint(-INFINITY);
      }
      float mx8[8];
#pragma unroll
      for (int a = 0; a < 8; ++a) mx8[a] = __uint_as_float(sr[a]);
#pragma unroll
      for (int i = 8; i < 64; ++i) mx8[i & 7] = fmaxf(mx8[i & 7], __uint_as_float(sr[i]));
      float mx = fmaxf(fmaxf(fmaxf(mx8[0], mx8[1]), fmaxf(mx8[2], mx8[3])),
                       fmaxf(fmaxf(mx8[4], mx8[5]), fmaxf(mx8[6], mx8[7])));
      sm.xch[half][row] = mx;
      named_bar_sync(pair_bar, 64);
      mx = fmaxf(mx, sm.xch[half ^ 1][row]);
      const float mnew = mx * c;
      float alpha = 1.f;
      const bool need = mnew > m_used + RESCALE_LOG2;
      if (need) {
        alpha = ex2(m_used - mnew);  // 0 on the first tile (m_used = -inf)
        l *= alpha;
        m_used = mnew;
      }
      const float neg = -m_used;
      uint32_t pk[32];
      float ls[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 32; ++i) {
        const float p0 = ex2(fmaf(__uint_as_float(sr[2 * i]), c, neg));
        const float p1 = ex2(fmaf(__uint_as_float(sr[2 * i + 1]), c, neg));
        ls[i & 3] += p0 + p1;
        pk[i] = pack_bf16x2(p0, p1);
      }
      l += (ls[0] + ls[1]) + (ls[2] + ls[3]);
      if (jj > 0) {
        // P V(it-1) must be done before P is overwritten and O is rescaled.
        mbar_wait(b_o, o_phase, abort_flag, WAIT_NS);
        o_phase ^= 1;
      }
      tc_fence_after();
      if (issuer && it >= 1) {
        // P V(it-1) has completed, so V(it-1)'s stage is free: refill it with
        // V(it+1) (V(0) and V(1) came with the prologue).
        if (x_begin + nv < x_end) {  // nv == it + VSTAGES - 1 here
          load_v(sm, p, &tmV, &tmBV, x_begin + nv, nv % VSTAGES);
          ++nv;
        }
      }
      tmem_st32(tmem + lane_off + p_col, pk);
      if (jj > 0 && __any_sync(0xffffffffu, need)) {
        uint32_t orr[32];
        tmem_ld32(tmem + lane_off + o_col, orr);
#pragma unroll
        for (int i = 0; i < 32; ++i) orr[i] = __float_as_uint(__uint_as_float(orr[i]) * alpha);
        tmem_st32(tmem + lane_off + o_col, orr);
      }
      tc_fence_before();
      __syncthreads();
      if (issuer) {
        tc_fence_after();
        const int sv = it % VSTAGES;
        if (mbar_wait(smem_addr(&sm.v_full[sv]), (it / VSTAGES) & 1, abort_flag, WAIT_NS)) {
          const uint32_t vaddr = smem_addr(sm.v[sv]);
#pragma unroll
          for (int kk = 0; kk < BN / 16; ++kk)
            mma_ts(tmem + TM_O, tmem + TM_P + kk * 8, sdesc_sw128(vaddr + kk * 2048), IDESC_PV,
                   (jj > 0 || kk > 0) ? 1u : 0u);
        }
        mma_commit(b_o);
      }
    }
    if (stop) break;
    // ------------------------------------------------------------ epilogue
    const bool ok = mbar_wait(b_o, o_phase, abort_flag, WAIT_NS);
    o_phase ^= 1;
    tc_fence_before();
    sm.xch[half][row] = l;
    if (__syncthreads_or(!ok || *abort_flag)) {
      stop = true;
      break;
    }
    tc_fence_after();
    const float lrow = l + sm.xch[half ^ 1][row];
    uint32_t orr[32];
    tmem_ld32(tmem + lane_off + o_col, orr);
    const float inv_l = 1.f / lrow;
    const float lse_val = (m_used + __log2f(lrow)) * 0.69314718055994531f;
    const int q = qt * BM + row;
    if (j0 == 0 && j1 == nkv) {
      if (q < p.N) {
        uint4* dst = reinterpret_cast<uint4*>(p.out + ((size_t)q * p.H + h) * HD + 32 * half);
#pragma unroll
        for (int c8 = 0; c8 < 4; ++c8) {
          uint4 w;
          w.x = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 0]) * inv_l, __uint_as_float(orr[c8 * 8 + 1]) * inv_l);
          w.y = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 2]) * inv_l, __uint_as_float(orr[c8 * 8 + 3]) * inv_l);
          w.z = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 4]) * inv_l, __uint_as_float(orr[c8 * 8 + 5]) * inv_l);
          w.w = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 6]) * inv_l, __uint_as_float(orr[c8 * 8 + 7]) * inv_l);
          dst[c8] = w;
        }
        if (half == 0) p.lse[(size_t)h * p.N + q] = lse_val;
      }
    } else {
      const int slot = (u == u_first) ? 0 : 1;
      const size_t pr = ((size_t)b * 2 + slot) * BM + row;
      float4* dst = reinterpret_cast<float4*>(p.part_o + pr * HD + 32 * half);
#pragma unroll
      for (int c4 = 0; c4 < 8; ++c4)
        dst[c4] = make_float4(__uint_as_float(orr[c4 * 4 + 0]) * inv_l, __uint_as_float(orr[c4 * 4 + 1]) * inv_l,
                              __uint_as_float(orr[c4 * 4 + 2]) * inv_l, __uint_as_float(orr[c4 * 4 + 3]) * inv_l);
      if (half == 0) p.part_lse[pr] = lse_val;
    }
    x += n;
    ++piece;
  }
  if (issuer) {
    // All MMAs issued have finished and every issued copy has landed before
    // shared memory and TMEM are released (matters only after an abort).
    mma_commit(b_fin);
    mbar_wait(b_fin, 0, never, DRAIN_NS);
    // the last load into a stage is the only one possibly still in flight
    for (int i = nk - KSTAGES > 0 ? nk - KSTAGES : 0; i < nk; ++i)
      mbar_wait(smem_addr(&sm.k_full[i % KSTAGES]), (i / KSTAGES) & 1, never, DRAIN_NS);
    for (int i = nv - VSTAGES > 0 ? nv - VSTAGES : 0; i < nv; ++i)
      mbar_wait(smem_addr(&sm.v_full[i % VSTAGES]), (i / VSTAGES) & 1, never, DRAIN_NS);
    if (q_issued > 0) mbar_wait(b_qfull, (q_issued - 1) & 1, never, DRAIN_NS);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(p.status, kStatusTimeout);
}

// Merges the partial (O_p, LSE_p) of every unit whose key tiles were split
// across CTAs:  LSE = log sum_p exp(LSE_p),  O = sum_p exp(LSE_p - LSE) O_p.
__global__ void __launch_bounds__(128) attn_combine_kernel(Params p, int G) {
  const int u = blockIdx.x;
  const long long T = p.total;
  const int nkv = p.nkv;
  auto cta_of = [&](long long x) {
    long long bb = x * G / T;
    while (bb + 1 < G && range_begin((int)bb + 1, G, T) <= x) ++bb;
    while (bb > 0 && range_begin((int)bb, G, T) > x) --bb;
    return (int)bb;
  };
  const int b_lo = cta_of((long long)u * nkv), b_hi = cta_of((long long)u * nkv + nkv - 1);
  if (b_lo == b_hi) return;  // finished inside one CTA
  const int h = u / p.nqt, qt = u - h * p.nqt;
  const int row = threadIdx.x;
  const int q = qt * BM + row;
  if (q >= p.N) return;
  float mx = -INFINITY;
  for (int bb = b_lo; bb <= b_hi; ++bb) {
    const int slot = (u == (int)(range_begin(bb, G, T) / nkv)) ? 0 : 1;
    mx = fmaxf(mx, p.part_lse[((size_t)bb * 2 + slot) * BM + row]);
  }
  float den = 0.f;
  for (int bb = b_lo; bb <= b_hi; ++bb) {
    const int slot = (u == (int)(range_begin(bb, G, T) / nkv)) ? 0 : 1;
    den += __expf(p.part_lse[((size_t)bb * 2 + slot) * BM + row] - mx);
  }
  const float lse = mx + __logf(den);
  float acc[HD];
#pragma unroll
  for (int i = 0; i < HD; ++i) acc[i] = 0.f;
  for (int bb = b_lo; bb <= b_hi; ++bb) {
    const int slot = (u == (int)(range_begin(bb, G, T) / nkv)) ? 0 : 1;
    const size_t pr = ((size_t)bb * 2 + slot) * BM + row;
    const float w = __expf(p.part_lse[pr] - lse);
    const float4* src = reinterpret_cast<const float4*>(p.part_o + pr * HD);
#pragma unroll
    for (int c4 = 0; c4 < 16; ++c4) {
      const float4 v = src[c4];
      acc[c4 * 4 + 0] += w * v.x;
      acc[c4 * 4 + 1] += w * v.y;
      acc[c4 * 4 + 2] += w * v.z;
      acc[c4 * 4 + 3] += w * v.w;
    }
  }
  uint4* dst = reinterpret_cast<uint4*>(p.out + ((size_t)q * p.H + h) * HD);
#pragma unroll
  for (int c8 = 0; c8 < 8; ++c8) {
    uint4 w;
    w.x = pack_bf16x2(acc[c8 * 8 + 0], acc[c8 * 8 + 1]);
    w.y = pack_bf16x2(acc[c8 * 8 + 2], acc[c8 * 8 + 3]);
    w.z = pack_bf16x2(acc[c8 * 8 + 4], acc[c8 * 8 + 5]);
    w.w = pack_bf16x2(acc[c8 * 8 + 6], acc[c8 * 8 + 7]);
    dst[c8] = w;
  }
  p.lse[(size_t)h * p.N + q] = lse;
}

}  // namespace

cudaError_t attn_setup() {
  cudaError_t e = cudaFuncSetAttribute(attn_fwd_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(attn_fwd_kernel, cudaFuncAttributePreferredSharedMemoryCarveout, 100);
}

int attn_ctas_per_sm() {
  int n = 0;
  if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, attn_fwd_kernel, THREADS, SMEM_BYTES) !=
      cudaSuccess)
    return 1;
  return n < 1 ? 1 : n;
}

int attn_smem_bytes() { return (int)SMEM_BYTES; }

cudaError_t launch_attention(const AttnArgs& a, bool combine, cudaStream_t s, cudaEvent_t ev_before,
                             cudaEvent_t ev_after) {
  Params p;
  p.N = a.N;
  p.H = a.H;
  p.M = a.M;
  p.nb = (a.M + BN - 1) / BN;
  const int nf = (a.N + BN - 1) / BN;
  p.nkv = p.nb + nf;
  p.nqt = (a.N + BM - 1) / BM;
  p.total = (long long)a.H * p.nqt * p.nkv;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.out = a.out;
  p.lse = a.lse;
  p.part_o = a.part_o;
  p.part_lse = a.part_lse;
  p.status = a.status;
  if (a.grid < 1 || (long long)a.grid > p.total) return cudaErrorInvalidValue;
  cudaError_t e;
  if (ev_before && (e = cudaEventRecord(ev_before, s)) != cudaSuccess) return e;
  attn_fwd_kernel<<<a.grid, THREADS, SMEM_BYTES, s>>>(*a.tmQ, *a.tmK, *a.tmV, *a.tmBK, *a.tmBV, p);
  e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  if (ev_after && (e = cudaEventRecord(ev_after, s)) != cudaSuccess) return e;
  if (!combine) return cudaSuccess;
  attn_combine_kernel<<<a.H * p.nqt, 128, 0, s>>>(p, a.grid);
  return cudaGetLastError();
}

}  // namespace regmem_dev
