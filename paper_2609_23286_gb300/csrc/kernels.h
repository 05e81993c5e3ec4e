// Internal launch interface between the C-ABI layer (regmem_api.cu) and the
// kernels.  Nothing here is exported from the shared library.
#pragma once

#include <cuda.h>
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <cstdint>

namespace regmem_dev {

// Launches `kernel` with programmatic stream serialization: it may start
// while the previous kernel in the stream finishes, and waits for it inside
// (griddepcontrol.wait) before touching what that kernel may read or write.
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                              cudaStream_t s, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args&&>(args)...);
}

constexpr int kHeadDim = 64;    // channels per head handled by the kernels
constexpr int kTile = 128;      // query rows / key rows per tile

// Bits of the device status word (written by kernels, read by the host).
constexpr int kStatusTimeout = 1;    // a bounded wait expired
constexpr int kStatusSmemAlign = 2;  // dynamic shared memory not 1 KB aligned
constexpr int kStatusRange = 4;      // a range guard of the checked build failed

// Range guards of the checked build (compiled with REGMEM_DEVICE_CHECKS, as
// libregmem_checked.so): an index a kernel derives before a global access
// is checked against its buffer; a failed check records kStatusRange in the
// status word and the access is skipped.  In the normal build dev_check is
// `true` and compiles away.
#ifdef REGMEM_DEVICE_CHECKS
constexpr bool kDeviceChecks = true;
#else
constexpr bool kDeviceChecks = false;
#endif
__device__ __forceinline__ bool dev_check(bool ok, int* status) {
  if constexpr (kDeviceChecks) {
    if (!ok) {
      atomicOr(status, kStatusRange);
      return false;
    }
  }
  return true;
}

// Largest attention grid: the merge of split units lists at most this many
// pieces per unit.
constexpr int kAttnMaxGrid = 256;

// The attention's stream-K split.  The (unit, key tile) sequence runs in P
// phases (P = 1 or 2), each a contiguous run of whole head-pair groups of
// units; CTA b takes key tiles [x[p][b], x[p][b + 1]) of phase p, phase by
// phase.  With two phases only half of the heads' K/V is read at any time:
// a long bank that L2 cannot hold whole (16 heads x 29,360 rows = 120 MB
// at the 2000-frame stream's end) is otherwise re-read ~4x from HBM,
// because the CTAs sweep every head's rows at scattered positions at once.
//
// The cuts equalise an estimated cost, not the tile count: a frame tile
// (the frame's own K/V, gathered from the token-major frame tensor, the last
// one ragged) costs more than a bank tile, and every unit a CTA starts costs
// a pipeline drain and refill.  The weights are per-CTA timings of the
// kernel at 16.7k keys regressed on these counts (a unit start ~1.7 tiles, a
// frame tile ~1.08).
constexpr int kCostBankTile = 100, kCostFrameTile = 108, kCostUnitStart = 170;
constexpr int kAttnMaxPhases = 2;
// K/V bytes of a launch above which it runs in two phases.
constexpr long long kAttnPhaseKvBytes = 80ll << 20;
struct SplitBounds {
  int P;                                          // phases
  int slots;                                      // partial slots per CTA (2 x the phases allowed)
  long long pbeg[kAttnMaxPhases + 1];             // first tile of each phase; pbeg[P] = total
  long long x[kAttnMaxPhases][kAttnMaxGrid + 1];  // the cuts of each phase
};
// Cuts units [u0, u1) (nb bank tiles then nf frame tiles each) into G ranges
// of about equal cost, into x[0..G]: strictly increasing, x[0] = u0 (nb +
// nf), x[G] = u1 (nb + nf).  Needs (u1 - u0) (nb + nf) >= G.
inline void attn_cut_phase(long long* x, long long u0, long long u1, int nb, int nf, int G) {
  const long long nkv = nb + nf, t0 = u0 * nkv, t1 = u1 * nkv;
  const long long wu = kCostUnitStart + (long long)kCostBankTile * nb + (long long)kCostFrameTile * nf;
  const long long wt = (u1 - u0) * wu;
  for (int b = 0; b <= G; ++b) {
    const long long target = wt / G * b + (wt % G) * b / G;  // floor(wt b / G) without overflow
    const long long u = target / wu;
    long long r = target - u * wu - kCostUnitStart, j;
    if (r <= 0) j = 0;
    else if (r < (long long)kCostBankTile * nb) j = (r + kCostBankTile / 2) / kCostBankTile;
    else j = nb + (r - (long long)kCostBankTile * nb + kCostFrameTile / 2) / kCostFrameTile;
    x[b] = t0 + u * nkv + (j < nkv ? j : nkv);
  }
  x[0] = t0;
  x[G] = t1;
  for (int b = 1; b < G; ++b)  // every CTA at least one tile
    if (x[b] <= x[b - 1]) x[b] = x[b - 1] + 1;
  for (int b = G - 1; b > 0; --b)
    if (x[b] > t1 - (G - b)) x[b] = t1 - (G - b);
}
// The split of `units` units (H heads, nqt query tiles per head; unit order
// of unit_tiles) over G CTAs: two phases when the K/V of the launch
// (H M 256 bytes) exceed kAttnPhaseKvBytes, there are at least two
// head-pair groups, max_phases allows it and each phase has at least G
// tiles; one phase otherwise.
inline void attn_split_bounds(SplitBounds& sb, long long units, int nb, int nf, int G, int H,
                              int nqt, long long M, int max_phases) {
  const long long nkv = nb + nf, total = units * nkv;
  const long long gs = 2 * (nqt >> 1) + (nqt & 1);  // units of a two-head group
  const long long ngroups = (H + 1) / 2;
  sb.P = 1;
  sb.slots = 2 * (max_phases > 1 ? kAttnMaxPhases : 1);
  sb.pbeg[0] = 0;
  if (max_phases > 1 && ngroups >= 2 && (long long)H * M * 256 > kAttnPhaseKvBytes) {
    const long long u1 = ((ngroups + 1) / 2) * gs;  // whole two-head groups in phase 0
    if (u1 * nkv >= G && (units - u1) * nkv >= G) {
      sb.P = 2;
      sb.pbeg[1] = u1 * nkv;
      sb.pbeg[2] = total;
      attn_cut_phase(sb.x[0], 0, u1, nb, nf, G);
      attn_cut_phase(sb.x[1], u1, units, nb, nf, G);
      return;
    }
  }
  sb.pbeg[1] = total;
  attn_cut_phase(sb.x[0], 0, units, nb, nf, G);
}

// The split as the merge of split units needs it (split.cuh).
struct SplitLayout {
  SplitBounds bnd;
  long long total;        // units * nkv
  int G;                  // attention CTAs
  int nkv;                // key tiles per unit
  int nqt;                // query tiles per head
  int N, H;
  const __nv_bfloat16* part_o;  // [G][bnd.slots][kUnitRows][64] piece partials (bf16)
  const float* part_lse;  // [G][bnd.slots][kUnitRows]
  __nv_bfloat16* out;     // [N][H][64]
  float* lse;             // [H][N]
  int* status;            // device status word (range guards of the checked build)
};

struct AttnArgs {
  const CUtensorMap* tmQ;   // frame tensors [N][H][64] bf16, box 64x1x128
  const CUtensorMap* tmK;
  const CUtensorMap* tmV;
  const CUtensorMap* tmBK;  // bank [H][cap][64] bf16, box 64x128x1
  const CUtensorMap* tmBV;
  int N, H, M;              // frame tokens, heads, bank rows per head
  float scale;
  __nv_bfloat16* out;       // [N][H][64]
  float* lse;               // [H][N]
  __nv_bfloat16* part_o;    // [grid][2 max_phases][kUnitRows][64] split-piece partials (bf16)
  float* part_lse;          // [grid][2 max_phases][kUnitRows]
  int max_phases;           // 1 or 2 (kAttnMaxPhases): phases the partial scratch allows
  int* status;
  int grid;                 // CTAs of the attention kernel (<= plan.total)
  // optional launch clock (nullptr: off), this launch's words, global timer
  // in ns: the earliest CTA start after the dependency wait (preset to ~0)
  // and the latest CTA end (preset to 0)
  unsigned long long* clk_start;
  unsigned long long* clk_end;
  // limit of every bounded wait in the kernel (ns; 2 s in normal use)
  unsigned long long wait_ns;
  // failure-detection tests only: CTA 0's producer does not issue this K/V
  // load (CTA-local load index), so the bounded waits on its stage run out;
  // -1 in normal use
  int fault_skip_kv;
};

// Work decomposition: a unit is a pair of 128-row query tiles run over all
// key tiles of [bank ; frame]: two consecutive tiles of one head, or, when a
// head has an odd number of query tiles, the last (lone) tiles of heads 2g
// and 2g + 1 together (a lone tile's softmax warpgroup paces its chain alone
// and leaves the tensor core idle half the time; paired, the two tiles keep
// it busy as a same-head pair does, at the cost of loading both heads' K/V).
// With an odd head count the last head's lone tile stays a unit by itself.
// Units are ordered by pairs of heads: head 2g's pairs, head 2g + 1's pairs,
// then their lone tiles, so units that read the same K/V run close in time.
constexpr int kUnitRows = 2 * kTile;
struct UnitTiles {
  int h0, qt0;  // head and query tile of the unit's first tile
  int h1, qt1;  // of its second tile (qt1 = qt0 + 1 past the last tile when has1 is false)
  bool has1;    // the second tile holds rows
};
__host__ __device__ inline long long attn_units(int nqt, int H) {
  return (long long)H * (nqt >> 1) + ((nqt & 1) ? (H + 1) / 2 : 0);
}
__host__ __device__ inline UnitTiles unit_tiles(long long u, int nqt, int H) {
  const int nfp = nqt >> 1, odd = nqt & 1;
  const int gs = 2 * nfp + odd;  // units of a group of two heads
  const int g = (int)(u / gs), r = (int)(u - (long long)g * gs);
  const bool two = 2 * g + 1 < H;  // the group has two heads (else: the last head alone)
  UnitTiles ut;
  ut.has1 = true;
  if (r < nfp || (two && r < 2 * nfp)) {  // a same-head pair
    ut.h0 = ut.h1 = 2 * g + (r >= nfp ? 1 : 0);
    ut.qt0 = 2 * (r >= nfp ? r - nfp : r);
    ut.qt1 = ut.qt0 + 1;
  } else if (two) {  // the lone tiles of heads 2g and 2g + 1
    ut.h0 = 2 * g;
    ut.h1 = 2 * g + 1;
    ut.qt0 = ut.qt1 = nqt - 1;
  } else {  // the last head's lone tile (odd head count)
    ut.h0 = ut.h1 = 2 * g;
    ut.qt0 = nqt - 1;
    ut.qt1 = nqt;
    ut.has1 = false;
  }
  return ut;
}
struct AttnPlan {
  long long units, tiles_per_unit, total;
};
AttnPlan attn_plan(int N, int H, int M);

// Scratch sizes for a given grid and phases allowed (two partial slots per
// CTA and phase: its first and its last piece).
inline size_t attn_part_o_elems(int grid, int max_phases) {
  return (size_t)grid * 2 * max_phases * kUnitRows * kHeadDim;
}
inline size_t attn_part_lse_floats(int grid, int max_phases) {
  return (size_t)grid * 2 * max_phases * kUnitRows;
}

// The split of an attention launch with these arguments.
SplitLayout attn_split_layout(const AttnArgs& a);
cudaError_t attn_setup();                              // kernel attributes (once)
int attn_ctas_per_sm();                                // resident CTAs per SM
int attn_smem_bytes();                                 // dynamic shared memory per CTA
// Launches the attention kernel and the merge of split units behind it;
// ev_before / ev_after (may be null) are recorded around the attention
// kernel, ev_merged after the merge.
cudaError_t launch_attention(const AttnArgs& a, cudaStream_t s, cudaEvent_t ev_before = nullptr,
                             cudaEvent_t ev_after = nullptr, cudaEvent_t ev_merged = nullptr);

// Per-head top-k of the candidates' saliency and append to the bank.
struct AdmitArgs {
  const float* sal;         // [H][N]
  const __nv_bfloat16* K;   // [N][H][64]
  const __nv_bfloat16* V;
  __nv_bfloat16* bankK;     // this layer's bank [H][cap][64]
  __nv_bfloat16* bankV;
  long long cap;
  long long M;              // rows already in the bank
  int N, H, cand_lo, k;
  int32_t* idx_out;         // optional [H][k]
  // distributed selection (k <= 32): per-(head, 128-key tile) lists and
  // completion counters (zero between launches): per head, or with `shared`
  // per key tile plus one for the tiles; null -> one block per head selects
  // alone
  uint64_t* lists;          // [H][ceil(N/128)][32]
  int* done;                // [max(H, ceil(N/128) + 1)]
  int* status;              // device status word (range guards of the checked build)
  int shared;               // fused path only: one token set for all heads (idx_out [k])
};
cudaError_t admit_setup();
// Per-head admission (Eq. 6): k rows per head, idx_out [H][k].
cudaError_t launch_admit(const AdmitArgs& a, cudaStream_t s);
// Admission without head-specific retention: one set of k tokens, ranked by
// the head sum of the saliency, appended to every head; idx_out [k].
cudaError_t launch_admit_shared(const AdmitArgs& a, cudaStream_t s);
// First frame (Eq. 4): bank[h][0:N] = frame rows of head h.
cudaError_t launch_anchor(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                          __nv_bfloat16* bankV, long long cap, int N, int H, int* status, cudaStream_t s);

// LSE-Saliency over the frame's own keys, per (head, 128-key tile).  With
// `adm` set (1 <= k <= 32, sal == adm->sal, lists and done given), each block
// also keeps its tile's best admission candidates and the last block to
// finish a head runs that head's admission.
struct SalArgs {
  const CUtensorMap* tmK;   // frame K map (same as the attention's)
  const __nv_bfloat16* Q;   // [N][H][64]
  const int* qidx;          // sampled query tokens, [nq]
  int nq;
  const float* lse;         // [H][N]
  int N, H;
  float scale;
  float* sal;               // [H][N]
  int* status;
  const AdmitArgs* adm;     // optional fused admission
};
cudaError_t saliency_setup();
cudaError_t launch_saliency(const SalArgs& a, cudaStream_t s);

constexpr int kMaxCandidates = 8192;
constexpr int kFusedMaxK = 32;  // largest k of the distributed (list) selection

}  // namespace regmem_dev
