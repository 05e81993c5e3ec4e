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
// Work split (stream-K over the key dimension): a unit is a pair of 128-row
// query tiles -- two consecutive tiles of one head, or the last tiles of two
// heads when a head has an odd number of them (unit_tiles) -- and the
// (unit, key tile) space is cut into `grid` contiguous ranges of about equal
// estimated cost, one per CTA (one CTA per SM; attn_split_bounds: a frame
// tile and the start of a unit cost more than a bank tile).  A unit whose
// key tiles all fall in one CTA is finished there (O in bf16 and LSE written
// directly).  A unit cut between CTAs leaves one normalised fp32 partial
// (O_p, LSE_p) per piece, in a slot of the CTA that computed it (its first or
// its last piece), and attn_combine_kernel, launched right behind, folds
// each split unit's pieces in CTA order,
//     LSE = log sum_p exp(LSE_p),  O = sum_p exp(LSE_p - LSE) O_p.
// No CTA waits for another.
// The kernel may start while its predecessor in the stream finishes: barrier
// setup and the TMEM allocation run before griddepcontrol.wait, everything
// that reads inputs or writes outputs after it.
//
// CTA layout, warp-specialised (12 warps, three warpgroups):
//   warp 0       TMA producer: both Q tiles of a unit, then K and V tiles
//                through a 6-stage ring (a stage holds one K and one V tile,
//                which land on one barrier; a two-head unit takes two stages
//                per key tile, one per head)
//   warp 1       Q K^T issuer (one lane) for both query tiles; owns TMEM
//   warps 2, 3   P V issuers (one lane each) for query tile 0 and 1
// The control warpgroup (warps 0-3) hands most of its register budget to
// the softmax warpgroups.
//   warps 4..7   softmax warpgroup 0 -> query tile 0 of the unit
//   warps 8..11  softmax warpgroup 1 -> query tile 1 of the unit
// Each softmax thread owns one query row (its TMEM lane).  Each key tile is
// loaded once and serves both query tiles (once per head for a two-head
// unit: each tile reads its own head's stage, and the other tile's P V
// issuer releases that stage with a plain arrival).
// TMEM (512 columns): S0 [0,128), S1 [128,256) fp32 logits; P0 [256,320),
// P1 [320,384) bf16 probabilities packed two per column; O0 [384,448),
// O1 [448,512) fp32 accumulators.  Q K^T is an SS-MMA (Q, K K-major in smem);
// P V is a TS-MMA (P from TMEM, V MN-major in smem).  Keeping P in TMEM keeps
// it off shared memory, whose bandwidth the SS-MMA operand reads and the TMA
// writes already use up.
// Hand-offs are mbarriers, per query tile: s_full (S(j) computed), s_free
// (S(j) read into registers), p_ready (P(j) stored), o_done (P V(j) done);
// plus the K/V ring's full/empty barriers (the empty ones take one arrival
// from each issuer) and Q full/empty.  On GB300 every mbarrier hand-off costs
// a few hundred cycles of latency, so the design keeps them off the critical
// chain where it can: the softmax releases S as soon as it holds S(j) in
// registers, and the Q K^T issuer computes S(j+1) while the softmax works on
// tile j; P is single-buffered, so the softmax waits for P V(j-1) (its
// o_done phase) before storing P(j).  The P V issuer never waits for its
// MMAs to complete: it commits each P V to o_done and moves on to the next
// p_ready, so P V(j) is issued as soon as P(j) is stored (measured 1 %
// shorter launches than an issuer that waited for each P V and published
// its completion in a shared word).
// With separate issuers for Q K^T and for each tile's P V, a Q K^T is never
// queued behind the issue of a P V in the same thread (an MMA issue blocks
// while the tensor core is busy), and one tile's P V never waits for the
// other tile's softmax.
// The softmax uses packed fp32x2 FMA/ADD and three-input max, leaving the
// exp2 (MUFU) as the dominant instruction stream.
// The softmax keeps a stale running max and only rescales O when the max
// grows by more than 2^8, so exp values stay <= 256.
// Every wait is bounded: on expiry a shared abort word stops all roles, the
// issued copies and MMAs are drained, TMEM is freed and a status bit is set.

#include "kernels.h"
#include "ptx.cuh"
#include "split.cuh"

namespace regmem_dev {
using namespace ptx;

namespace {

constexpr int BM = kTile, BN = kTile, HD = kHeadDim;
constexpr int UROWS = kUnitRows;         // query rows per unit (two tiles)
constexpr int STAGES = 6;  // K/V ring depth (a stage holds one K tile and one V tile)
constexpr int TILE_BYTES = BM * HD * 2;  // 16 KB bf16 tile
constexpr int THREADS = 384;
// Register split: launched at 168 per thread (384 x 168 = 64,512); the
// control warpgroup drops to 56 and the two softmax warpgroups rise to 224,
// 128 x 56 + 256 x 224 = 64,512, the launch total.
constexpr uint32_t REGS_CTRL = 56, REGS_SOFTMAX = 224;
static_assert(128 * REGS_CTRL + 256 * REGS_SOFTMAX <= THREADS * 168, "register split");
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t TM_S0 = 0, TM_S1 = 128, TM_P0 = 256, TM_P1 = 320, TM_O0 = 384, TM_O1 = 448;
constexpr uint64_t DRAIN_NS = 200000000ull;   // 0.2 s for draining on abort
constexpr float RESCALE_LOG2 = 8.0f;
constexpr uint32_t IDESC_QK = idesc_bf16_f32(128, 128, false, false);
constexpr uint32_t IDESC_PV = idesc_bf16_f32(128, 64, false, true);

struct Smem {
  uint8_t q[2][TILE_BYTES];
  uint8_t k[STAGES][TILE_BYTES];
  uint8_t v[STAGES][TILE_BYTES];
  uint64_t q_full, q_empty;
  uint64_t kv_full[STAGES], kv_empty[STAGES];
  uint64_t s_full[2], s_free[2], p_ready[2], o_done[2];  // per query tile
  uint64_t fin_bar;
  uint32_t tmem_base;
  int abort_flag;
  int never;  // always 0: abort word for waits that must not be cut short
};
// The dynamic shared window is requested 1 KB aligned (128-byte swizzle
// atoms need it) and checked at run time.
constexpr size_t SMEM_BYTES = (sizeof(Smem) + 127) & ~size_t(127);
static_assert(SMEM_BYTES <= 232448, "more dynamic shared memory than a CTA can have (227 KB)");

struct Params {
  SplitBounds bnd;  // this launch's split: CTA b takes tiles [bnd.x[p][b], bnd.x[p][b + 1]) of phase p
  int N, H, M;
  int nb, nkv, nqt;
  long long total;
  float scale_log2;
  __nv_bfloat16* out;
  float* lse;
  __nv_bfloat16* part_o;  // [grid][bnd.slots][256][64]: partials of each CTA's first / last
                          // piece of each phase
  float* part_lse;  // [grid][bnd.slots][256]
  int* status;
  unsigned long long* clk_start;  // launch clock (AttnArgs) or nullptr
  unsigned long long* clk_end;
  unsigned long long wait_ns;     // limit of every bounded wait (AttnArgs)
  int fault_skip_kv;              // failure-detection tests: CTA 0 skips this K/V load
};


__device__ __forceinline__ int tile_valid(const Params& p, int j) {
  return j < p.nb ? min(BN, p.M - j * BN) : min(BN, p.N - (j - p.nb) * BN);
}

// One piece of a CTA's range: unit u, key tiles [j0, j1).
struct Piece {
  int u, j0, j1;
  UnitTiles ut;  // the unit's two query tiles (head, tile index)
  int kvs;       // K/V stages per key tile: 2 when the tiles belong to two heads
};
__device__ __forceinline__ Piece piece_at(const Params& p, long long x, long long x_end) {
  Piece pc;
  pc.u = (int)(x / p.nkv);
  pc.j0 = (int)(x - (long long)pc.u * p.nkv);
  pc.j1 = (int)min((long long)p.nkv, pc.j0 + (x_end - x));
  pc.ut = unit_tiles(pc.u, p.nqt, p.H);
  pc.kvs = pc.ut.h0 != pc.ut.h1 ? 2 : 1;
  return pc;
}

__global__ void __launch_bounds__(THREADS, 1)
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

  const int G = gridDim.x, b = blockIdx.x;

  if (tid == 0) {
    sm.abort_flag = 0;
    sm.never = 0;
    mbar_init(smem_addr(&sm.q_full), 1);
    mbar_init(smem_addr(&sm.q_empty), 1);
    for (int s = 0; s < STAGES; ++s) {
      mbar_init(smem_addr(&sm.kv_full[s]), 1);
      mbar_init(smem_addr(&sm.kv_empty[s]), 3);  // one arrival per issuer
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(smem_addr(&sm.s_full[t]), 1);
      mbar_init(smem_addr(&sm.s_free[t]), BM);   // every softmax thread arrives
      mbar_init(smem_addr(&sm.p_ready[t]), BM);
      mbar_init(smem_addr(&sm.o_done[t]), 1);
    }
    mbar_init(smem_addr(&sm.fin_bar), 3);
    fence_barrier_init();
  }
  if (warp == 1) {
    tmem_alloc(smem_addr(&sm.tmem_base), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  grid_dep_wait();  // the previous kernel's writes are visible, its reads done
  if (p.clk_start && tid == 0) atomicMin(p.clk_start, globaltimer_ns());

  if (warp < 4) {
   setmaxnreg_dec<REGS_CTRL>();
   if (warp == 0) {
    // ================================================================ producer
    if (lane == 0) {
      prefetch_tmap(&tmQ);
      prefetch_tmap(&tmK);
      prefetch_tmap(&tmV);
      prefetch_tmap(&tmBK);
      prefetch_tmap(&tmBV);
      int nkv = 0, piece = 0;  // K/V tile pairs, Q pairs issued
      bool ok = true;
      for (int ph = 0; ph < p.bnd.P && ok; ++ph) {
        const long long x_begin = p.bnd.x[ph][b], x_end = p.bnd.x[ph][b + 1];
        for (long long x = x_begin; x < x_end && ok;) {
          const Piece pc = piece_at(p, x, x_end);
          if (piece > 0) ok = mbar_wait(smem_addr(&sm.q_empty), (piece - 1) & 1, abort_flag, p.wait_ns);
          if (!ok) break;
          const uint32_t bq = smem_addr(&sm.q_full);
          mbar_arrive_expect_tx(bq, 2 * TILE_BYTES);
          // (a unit without a second tile loads rows past the frame: zero fill)
          tma_load_3d(smem_addr(sm.q[0]), &tmQ, bq, 0, pc.ut.h0, pc.ut.qt0 * BM);
          tma_load_3d(smem_addr(sm.q[1]), &tmQ, bq, 0, pc.ut.h1, pc.ut.qt1 * BM);
          ++piece;
          for (int j = pc.j0; j < pc.j1 && ok; ++j) {
            for (int hs = 0; hs < pc.kvs && ok; ++hs) {  // one stage per head of the unit
              const int st = nkv % STAGES, h = hs ? pc.ut.h1 : pc.ut.h0;
              if (nkv >= STAGES)
                ok = mbar_wait(smem_addr(&sm.kv_empty[st]), ((nkv / STAGES) - 1) & 1, abort_flag, p.wait_ns);
              if (!ok) break;
              // K and V of the tile land on one barrier: the issuer waits once
              const uint32_t bkv = smem_addr(&sm.kv_full[st]);
              if (b == 0 && nkv == p.fault_skip_kv) {  // injected fault: nothing lands here
                ++nkv;
                continue;
              }
              mbar_arrive_expect_tx(bkv, 2 * TILE_BYTES);
              if (j < p.nb) {
                tma_load_3d(smem_addr(sm.k[st]), &tmBK, bkv, 0, j * BN, h);
                tma_load_3d(smem_addr(sm.v[st]), &tmBV, bkv, 0, j * BN, h);
              } else {
                tma_load_3d(smem_addr(sm.k[st]), &tmK, bkv, 0, h, (j - p.nb) * BN);
                tma_load_3d(smem_addr(sm.v[st]), &tmV, bkv, 0, h, (j - p.nb) * BN);
              }
              ++nkv;
            }
          }
          x += pc.j1 - pc.j0;
        }
      }
      // Every issued copy must land before the CTA exits; the last load into
      // each stage is the only one that can still be in flight.
      for (int i = nkv - STAGES > 0 ? nkv - STAGES : 0; i < nkv; ++i)
        if (!(b == 0 && i == p.fault_skip_kv))
          mbar_wait(smem_addr(&sm.kv_full[i % STAGES]), (i / STAGES) & 1, never, DRAIN_NS);
      if (piece > 0) mbar_wait(smem_addr(&sm.q_full), (piece - 1) & 1, never, DRAIN_NS);
    }
  } else {
    // ================================================================ MMA issuers
    // Warp 1 issues every Q K^T (both query tiles), warp 2 the P V of query
    // tile 0 and warp 3 that of tile 1, so a Q K^T never waits behind the
    // issue of a P V in the same thread, and neither P V issuer waits for the
    // other tile's softmax.  All walk the tiles of the CTA's range in order.
    if (lane == 0) {
      const bool qk_role = warp == 1;
      const int tpv = warp - 2;  // query tile of a P V issuer
      uint32_t ph0 = 0, ph1 = 0;  // s_free (QK) or p_ready (PV) phases consumed, per query tile
      int it = 0, piece = 0;
      bool ok = true;
      for (int ph = 0; ph < p.bnd.P && ok; ++ph) {
        const long long x_begin = p.bnd.x[ph][b], x_end = p.bnd.x[ph][b + 1];
        for (long long x = x_begin; x < x_end && ok;) {
          const Piece pc = piece_at(p, x, x_end);
          const int n = pc.j1 - pc.j0;
          x += n;
          ++piece;
          const int ntiles = pc.ut.has1 ? 2 : 1;  // query tiles of this unit
          // CTA-local stage use of key tile jj for query tile t: one stage per
          // key tile, or two (one per head) when the tiles belong to two heads
          const int t0 = it;
          it += n * pc.kvs;
          auto use_of = [&](int jj, int t) { return t0 + jj * pc.kvs + (pc.kvs == 2 ? t : 0); };
          if (qk_role) {
            // Q K^T(j) of query tile t goes out once S(j-1) of that tile has
            // been read; the Q tiles are released after the piece's last one,
            // each stage after the Q K^T of both tiles has read its K.
            ok = mbar_wait(smem_addr(&sm.q_full), (piece - 1) & 1, abort_flag, p.wait_ns);
            for (int jj = 0; jj < n && ok; ++jj) {
              for (int t = 0; t < ntiles && ok; ++t) {
                const int tq = use_of(jj, t), st = tq % STAGES;
                if (t == 0 || pc.kvs == 2) {  // the stage holding this tile's K
                  ok = mbar_wait(smem_addr(&sm.kv_full[st]), (tq / STAGES) & 1, abort_flag, p.wait_ns);
                  if (!ok) break;
                }
                if (jj > 0) {
                  ok = mbar_wait(smem_addr(&sm.s_free[t]), (t ? ph1 : ph0) & 1, abort_flag, p.wait_ns);
                  if (t) ++ph1; else ++ph0;
                  if (!ok) break;
                }
                tc_fence_after();
                const uint32_t sq = smem_addr(sm.q[t]), d_s = tmem + (t ? TM_S1 : TM_S0);
                const uint32_t kaddr = smem_addr(sm.k[st]);
  #pragma unroll
                for (int kk = 0; kk < HD / 16; ++kk)
                  mma_ss(d_s, sdesc_sw128(sq + kk * 32), sdesc_sw128(kaddr + kk * 32), IDESC_QK, kk > 0);
                mma_commit(smem_addr(&sm.s_full[t]));
                // the stage's K is read by the last Q K^T that uses it
                if (t == ntiles - 1 || pc.kvs == 2) mma_commit(smem_addr(&sm.kv_empty[st]));
              }
            }
            mma_commit(smem_addr(&sm.q_empty));
            // the softmax also arrives on s_free for the piece's last tile; the
            // next piece's first Q K^T waits for it
            if (ok) ok = mbar_wait(smem_addr(&sm.s_free[0]), ph0 & 1, abort_flag, p.wait_ns);
            ++ph0;
            if (ok && ntiles == 2) {
              ok = mbar_wait(smem_addr(&sm.s_free[1]), ph1 & 1, abort_flag, p.wait_ns);
              ++ph1;
            }
          } else if (tpv == 0 || pc.ut.has1) {
            // P V(j) of the query tile goes out once P(j) is stored; its
            // completion releases P (o_done, waited by the softmax) and the
            // stage (the last read of its V).  The issuer does not wait for it.
            const uint32_t b_pready = smem_addr(&sm.p_ready[tpv]), b_odone = smem_addr(&sm.o_done[tpv]);
            const uint32_t d_o = tmem + (tpv ? TM_O1 : TM_O0), d_p = tmem + (tpv ? TM_P1 : TM_P0);
            for (int jj = 0; jj < n && ok; ++jj) {
              const int st = use_of(jj, tpv) % STAGES;
              ok = mbar_wait(b_pready, ph0 & 1, abort_flag, p.wait_ns);
              ++ph0;
              if (!ok) break;
              tc_fence_after();
              const uint32_t vaddr = smem_addr(sm.v[st]);
  #pragma unroll
              for (int kk = 0; kk < BN / 16; ++kk)  // 16 keys = 8 packed columns of P
                mma_ts(d_o, d_p + kk * 8, sdesc_sw128(vaddr + kk * 2048), IDESC_PV,
                       (jj == 0 && kk == 0) ? 0u : 1u);
              mma_commit(b_odone);
              mma_commit(smem_addr(&sm.kv_empty[st]));
              if (ok && pc.kvs == 2) {
                // the other head's stage of this key tile: this issuer's release
                // of it (an arrival only after that use's load has landed)
                const int to = use_of(jj, 1 - tpv), so = to % STAGES;
                ok = mbar_wait(smem_addr(&sm.kv_full[so]), (to / STAGES) & 1, abort_flag, p.wait_ns);
                if (ok) mbar_arrive(smem_addr(&sm.kv_empty[so]));
              }
            }
          } else {
            // tile 1 of a unit without one: nothing to compute, but the stage
            // releases keep their order (an arrival for a stage's next use
            // only after that use's load has landed)
            for (int jj = 0; jj < n && ok; ++jj) {
              const int tq = use_of(jj, 0), st = tq % STAGES;
              ok = mbar_wait(smem_addr(&sm.kv_full[st]), (tq / STAGES) & 1, abort_flag, p.wait_ns);
              if (ok) mbar_arrive(smem_addr(&sm.kv_empty[st]));
            }
          }
        }
      }
      // all issued MMAs finish before TMEM and shared memory are released
      mma_commit(smem_addr(&sm.fin_bar));
      mbar_wait(smem_addr(&sm.fin_bar), 0, never, DRAIN_NS);
    }
   }
  } else {
    setmaxnreg_inc<REGS_SOFTMAX>();
    // ================================================================ softmax
    const int t = (warp - 4) >> 2;          // query tile of this warpgroup
    const int quarter = warp & 3;           // TMEM lane quarter of this warp
    const int row = quarter * 32 + lane;    // query row inside the tile
    const uint32_t lane_off = (uint32_t)(quarter * 32) << 16;
    const uint32_t tm_s = tmem + lane_off + (t ? TM_S1 : TM_S0);
    const uint32_t tm_o = tmem + lane_off + (t ? TM_O1 : TM_O0);
    const uint32_t b_sfull = smem_addr(&sm.s_full[t]), b_pready = smem_addr(&sm.p_ready[t]);
    const uint32_t b_sfree = smem_addr(&sm.s_free[t]), b_odone = smem_addr(&sm.o_done[t]);
    const uint32_t tm_p = tmem + lane_off + (t ? TM_P1 : TM_P0);
    const float c = p.scale_log2;
    uint32_t s_phase = 0, o_phase = 0;  // s_full parity, P V completions consumed
    bool stop = false;
    // Bounded wait for a barrier phase (gives up on the abort word or after
    // p.wait_ns); a warp stops as a whole if any of its lanes gave up.
    auto wait_phase = [&](uint32_t bar, uint32_t parity) -> bool {
      const bool ok = mbar_wait(bar, parity, abort_flag, p.wait_ns);
      if (__any_sync(0xffffffffu, !ok)) return false;
      tc_fence_after();
      return true;
    };
    // Per key tile the warpgroup waits for S(j), arrives on s_free once S(j)
    // is in registers, waits for P V(j-1) (P is single-buffered) before
    // storing P(j), and arrives on p_ready once P(j) is stored.  Every thread
    // arrives (cheaper than a warp-elected arrival after a warp barrier).
    for (int ph = 0; ph < p.bnd.P && !stop; ++ph) {
      const long long x_begin = p.bnd.x[ph][b], x_end = p.bnd.x[ph][b + 1];
      for (long long x = x_begin; x < x_end && !stop;) {
        const Piece pc = piece_at(p, x, x_end);
        const int n = pc.j1 - pc.j0;
        x += n;
        if (t == 1 && !pc.ut.has1) continue;  // no rows in this unit's second tile
        const int th = t ? pc.ut.h1 : pc.ut.h0, tqt = t ? pc.ut.qt1 : pc.ut.qt0;  // this tile's head, index
        float m_used = -INFINITY;  // running max of the logits, scaled to log2 units
        float l = 0.f;             // running row sum of exp2(z*c - m_used)
        for (int jj = 0; jj < n; ++jj) {
          const int j = pc.j0 + jj;
          if (!wait_phase(b_sfull, s_phase)) {  // S(j) in TMEM
            stop = true;
            break;
          }
          s_phase ^= 1;
          uint32_t sr[128];
          tmem_ld128(tm_s, sr);
          tc_fence_before();
          mbar_arrive(b_sfree);  // S may be overwritten by the next Q K^T
          const int valid = tile_valid(p, j);
          if (valid < BN) {
  #pragma unroll
            for (int i = 0; i < 128; ++i)
              if (i >= valid) sr[i] = __float_as_uint(-INFINITY);
          }
          // row max: four independent chains of three-input max
          float mx4[4];
  #pragma unroll
          for (int a = 0; a < 4; ++a) mx4[a] = __uint_as_float(sr[a]);
  #pragma unroll
          for (int i = 4; i < 124; i += 8) {
  #pragma unroll
            for (int a = 0; a < 4; ++a)
              mx4[a] = fmax3(mx4[a], __uint_as_float(sr[i + 2 * a]), __uint_as_float(sr[i + 2 * a + 1]));
          }
          mx4[0] = fmax3(mx4[0], __uint_as_float(sr[124]), __uint_as_float(sr[125]));
          mx4[1] = fmax3(mx4[1], __uint_as_float(sr[126]), __uint_as_float(sr[127]));
          const float mx = fmax3(mx4[0], mx4[1], fmaxf(mx4[2], mx4[3]));
          const float mnew = mx * c;
          float alpha = 1.f;
          const bool need = mnew > m_used + RESCALE_LOG2;
          if (need) {
            alpha = ex2(m_used - mnew);  // 0 on the first tile (m_used = -inf)
            l *= alpha;
            m_used = mnew;
          }
          // p = exp2(z * c - m_used): packed FMA for the argument, MUFU exp2,
          // packed ADD for the row sum, bf16x2 pack.  P is computed in registers
          // before its TMEM columns are known to be free.
          const uint64_t cc = f2_pack(c, c), nn = f2_pack(-m_used, -m_used);
          uint64_t acc2[2] = {f2_pack(0.f, 0.f), f2_pack(0.f, 0.f)};
          uint32_t pk[2][32];
  #pragma unroll
          for (int hf = 0; hf < 2; ++hf) {
  #pragma unroll
            for (int i = 0; i < 32; ++i) {
              const int e = hf * 64 + 2 * i;
              float a0, a1;
              f2_unpack(f2_fma(f2_pack(__uint_as_float(sr[e]), __uint_as_float(sr[e + 1])), cc, nn), a0, a1);
              const float p0 = ex2(a0), p1 = ex2(a1);
              acc2[i & 1] = f2_add(acc2[i & 1], f2_pack(p0, p1));
              pk[hf][i] = pack_bf16x2(p0, p1);
            }
          }
          if (jj > 0) {
            // P V(j-1) has read P and added into O (at most one P V of this
            // tile is outstanding here, so the parity is unambiguous)
            if (!wait_phase(b_odone, (o_phase++) & 1)) {
              stop = true;
              break;
            }
            if (__any_sync(0xffffffffu, need)) {
              // rare (the max grew by > 2^8): rescale O before P V(j) adds to it
  #pragma unroll 1
              for (int hc = 0; hc < 2; ++hc) {  // 32 columns at a time
                uint32_t orr[32];
                tmem_ld32(tm_o + 32 * hc, orr);
  #pragma unroll
                for (int i = 0; i < 32; ++i) orr[i] = __float_as_uint(__uint_as_float(orr[i]) * alpha);
                tmem_st32(tm_o + 32 * hc, orr);
              }
            }
          }
          tmem_st32_async(tm_p, pk[0]);
          tmem_st32_async(tm_p + 32, pk[1]);
          tmem_wait_st();
          tc_fence_before();
          mbar_arrive(b_pready);
          {
            float s0, s1, s2, s3;
            f2_unpack(acc2[0], s0, s1);
            f2_unpack(acc2[1], s2, s3);
            l += (s0 + s1) + (s2 + s3);
          }
        }
        if (stop) break;
        // -------------------------------------------------------------- epilogue
        if (!wait_phase(b_odone, (o_phase++) & 1)) {  // the last tile's P V
          stop = true;
          break;
        }
        uint32_t orr[64];
        tmem_ld64(tm_o, orr);
        tc_fence_before();
        const float inv_l = 1.f / l;
        const float lse_val = (m_used + __log2f(l)) * 0.69314718055994531f;
        const int q = tqt * BM + row;
        if (pc.j0 == 0 && pc.j1 == p.nkv) {
          if (q < p.N) {
            uint4* dst = reinterpret_cast<uint4*>(p.out + ((size_t)q * p.H + th) * HD);
  #pragma unroll
            for (int c8 = 0; c8 < 8; ++c8) {
              uint4 w;
              w.x = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 0]) * inv_l, __uint_as_float(orr[c8 * 8 + 1]) * inv_l);
              w.y = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 2]) * inv_l, __uint_as_float(orr[c8 * 8 + 3]) * inv_l);
              w.z = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 4]) * inv_l, __uint_as_float(orr[c8 * 8 + 5]) * inv_l);
              w.w = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 6]) * inv_l, __uint_as_float(orr[c8 * 8 + 7]) * inv_l);
              dst[c8] = w;
            }
            p.lse[(size_t)th * p.N + q] = lse_val;
          }
        } else {
          // a piece of a unit split between CTAs: its normalised partial goes
          // to the CTA's slot (0: the CTA's first piece, 1: its last piece);
          // attn_combine_kernel merges the unit's pieces
          const int which = (x - n == x_begin) ? 0 : 1;
          const size_t pr = ((size_t)b * p.bnd.slots + 2 * ph + which) * UROWS + t * BM + row;
          if (!dev_check(2 * ph + which < p.bnd.slots, p.status)) continue;
          // O_p in bf16 (half the bytes the merge reads back), LSE_p in fp32;
          // the LSE is kept in L2 (evict_last) until the merge reads it
          const uint64_t pol = l2_policy_evict_last();
          uint4* dst = reinterpret_cast<uint4*>(p.part_o + pr * HD);
  #pragma unroll
          for (int c8 = 0; c8 < 8; ++c8) {
            uint4 w;
            w.x = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 0]) * inv_l, __uint_as_float(orr[c8 * 8 + 1]) * inv_l);
            w.y = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 2]) * inv_l, __uint_as_float(orr[c8 * 8 + 3]) * inv_l);
            w.z = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 4]) * inv_l, __uint_as_float(orr[c8 * 8 + 5]) * inv_l);
            w.w = pack_bf16x2(__uint_as_float(orr[c8 * 8 + 6]) * inv_l, __uint_as_float(orr[c8 * 8 + 7]) * inv_l);
            dst[c8] = w;
          }
          st_global_hint(p.part_lse + pr, lse_val, pol);
        }
      }
    }
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 1) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(p.status, kStatusTimeout);
  // launch clock: fire-and-forget reductions, nothing waits for them
  if (p.clk_end && tid == 0) atomicMax(p.clk_end, globaltimer_ns());
  // The merge kernel behind is released only as CTAs finish: released at the
  // start, its small blocks took SMs as they freed up and held them while
  // waiting, which measured 25 us slower per launch.
  grid_dep_launch();
}

// Merges the pieces of every split unit (split.cuh): block b takes merge job
// jobs.j[b], tile j & 1 of the unit cut by the boundary between CTAs j / 2
// and j / 2 + 1.  Only the jobs that merge something are launched (the host
// lists them), at most 2 (G - 1) blocks, two per SM: every block is resident
// at once, and the SMs without a merge block are free for the next kernel.
constexpr int CMB_THREADS = 4 * BM;
struct CombineJobs {
  unsigned short j[2 * kAttnMaxPhases * kAttnMaxGrid];
};

__global__ void __launch_bounds__(CMB_THREADS, 2)
    attn_combine_kernel(const SplitLayout lay, const CombineJobs jobs) {
  const unsigned j = jobs.j[blockIdx.x];
  const split::Job jb = split::prepare_job(lay, j == 0xFFFFu ? -1 : (int)j);  // layout only: before the wait
  grid_dep_wait();  // every piece's partial is stored
  grid_dep_launch();
  split::run_job<CMB_THREADS>(lay, jb, threadIdx.x);
}

Params make_params(const AttnArgs& a) {
  Params p;
  {
    const int nb = (a.M + BN - 1) / BN, nf = (a.N + BN - 1) / BN;
    const long long units = attn_units((a.N + BM - 1) / BM, a.H);
    const long long total = units * (nb + nf);
    attn_split_bounds(p.bnd, units, nb, nf, (int)(a.grid < total ? a.grid : total), a.H,
                      (a.N + BM - 1) / BM, a.M, a.max_phases);
  }
  p.N = a.N;
  p.H = a.H;
  p.M = a.M;
  p.nb = (a.M + BN - 1) / BN;
  const int nf = (a.N + BN - 1) / BN;
  p.nkv = p.nb + nf;
  p.nqt = (a.N + BM - 1) / BM;
  p.total = attn_units(p.nqt, a.H) * p.nkv;
  p.scale_log2 = a.scale * 1.4426950408889634f;
  p.out = a.out;
  p.lse = a.lse;
  p.part_o = a.part_o;
  p.part_lse = a.part_lse;
  p.status = a.status;
  p.clk_start = a.clk_start;
  p.clk_end = a.clk_end;
  p.wait_ns = a.wait_ns;
  p.fault_skip_kv = a.fault_skip_kv;
  return p;
}

}  // namespace

SplitLayout attn_split_layout(const AttnArgs& a) {
  const Params p = make_params(a);
  SplitLayout l;
  l.bnd = p.bnd;
  l.total = p.total;
  l.G = a.grid;
  l.nkv = p.nkv;
  l.nqt = p.nqt;
  l.N = a.N;
  l.H = a.H;
  l.part_o = a.part_o;
  l.part_lse = a.part_lse;
  l.out = a.out;
  l.lse = a.lse;
  l.status = a.status;
  return l;
}

AttnPlan attn_plan(int N, int H, int M) {
  AttnPlan pl;
  pl.units = attn_units((N + BM - 1) / BM, H);
  pl.tiles_per_unit = (M + BN - 1) / BN + (N + BN - 1) / BN;
  pl.total = pl.units * pl.tiles_per_unit;
  return pl;
}

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

cudaError_t launch_attention(const AttnArgs& a, cudaStream_t s, cudaEvent_t ev_before,
                             cudaEvent_t ev_after, cudaEvent_t ev_merged) {
  const Params p = make_params(a);
  if (a.grid < 1 || a.grid > kAttnMaxGrid || (long long)a.grid > p.total) return cudaErrorInvalidValue;
  cudaError_t e;
  if (ev_before && (e = cudaEventRecord(ev_before, s)) != cudaSuccess) return e;
  e = launch_pdl(attn_fwd_kernel, dim3(a.grid), dim3(THREADS), SMEM_BYTES, s, *a.tmQ, *a.tmK, *a.tmV,
                 *a.tmBK, *a.tmBV, p);
  if (e != cudaSuccess) return e;
  if (ev_after && (e = cudaEventRecord(ev_after, s)) != cudaSuccess) return e;
  if (a.grid > 1) {  // with one CTA no unit is split
    const SplitLayout lay = attn_split_layout(a);
    CombineJobs jobs;
    unsigned n = 0;
    for (int j = 0; j < split::job_count(lay); ++j)
      if (split::job_live(lay, j)) jobs.j[n++] = (unsigned short)j;
    if (n == 0) jobs.j[n++] = 0xFFFF;  // one block that merges nothing: the launch is counted
    e = launch_pdl(attn_combine_kernel, dim3(n), dim3(CMB_THREADS), 0, s, lay, jobs);
    if (e != cudaSuccess) return e;
  }
  if (ev_merged && (e = cudaEventRecord(ev_merged, s)) != cudaSuccess) return e;
  return cudaSuccess;
}

}  // namespace regmem_dev
