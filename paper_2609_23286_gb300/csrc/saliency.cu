// LSE-Saliency (Sec. 3.3, "FlashAttention-Compatible Saliency Estimation" and
// "Head-Specific Token Retention"):
//     S_j = sum_{i in Q~} exp(Z_ij - LSE_i),  Z_ij = q_i k_j^T * scale,
// for the frame's own keys j, per head, with LSE_i the row log-sum-exp over the
// whole attended context (memory + frame) written by the attention kernel.
//
// One CTA per (head, 128-key tile).  The tensor core computes the transposed
// logits Z^T = K_tile Q~_chunk^T (M = 128 keys in TMEM lanes, N = 128 sampled
// queries in TMEM columns), so each thread owns one key and the column sum of
// the paper becomes a private sum over its row: no cross-thread reduction and
// a fixed summation order (deterministic).  exp is taken in fp32 on the exact
// fp32 logits, never on the bf16 P of the attention kernel.
// The key tile arrives by TMA while every thread gathers its sampled query
// rows with 16-byte cp.async copies into 128-byte-swizzled tiles; up to four
// 128-query chunks are resident at once, and all of a group's index and LSE
// loads are issued before any of the copies that depend on them.  Z^T
// alternates between two 128-column TMEM buffers: the MMA of chunk c+2 is
// issued as soon as every thread has read chunk c, so it runs under the
// exponentials of chunk c.
//
// Fused admission (Eq. 6): when the launch carries admission arguments, each
// block sorts its tile's candidates (select.cuh) and stores its best 32, then
// adds itself to its head's completion counter; the last block of a head
// merges the tiles' lists into the head's k admitted tokens, appends their K
// and V rows to the bank and clears the counter for the next launch.  With
// `shared` (no head-specific retention) the counters are per key tile: the
// last head of a tile ranks the head sums of its tokens, and the last tile
// merges the lists and appends the same rows to every head.

#include "kernels.h"
#include "ptx.cuh"
#include "select.cuh"

namespace regmem_dev {
using namespace ptx;

namespace {

constexpr int BT = kTile, HD = kHeadDim;
constexpr int TILE_BYTES = BT * HD * 2;
constexpr int THREADS = 128;
constexpr int QS = 4;                 // resident sampled-query chunks
constexpr uint32_t TMEM_COLS = 256;   // two 128-column Z^T buffers
constexpr uint64_t WAIT_NS = 2000000000ull;
constexpr uint64_t DRAIN_NS = 200000000ull;
constexpr uint32_t IDESC = idesc_bf16_f32(128, 128, false, false);
constexpr int MAX_CHUNKS = 64;  // sampled queries <= 8192

struct Smem {
  uint8_t k[TILE_BYTES];
  uint8_t qs[QS][TILE_BYTES];  // after the saliency: admission keys and positions
  float lse2[QS][BT];
  uint64_t k_full, mma_bar[2], fin_bar;
  uint32_t tmem_base;
  int abort_flag;
  int never;
  int last;                    // this block finished its head's saliency last
};
// About 83 KB: at most two CTAs share an SM, so their two 256-column TMEM
// allocations fit the SM's 512 columns.
constexpr size_t SMEM_BYTES = sizeof(Smem) + 1024;

struct Params {
  const __nv_bfloat16* Q;
  const int* qidx;
  int nq;
  const float* lse;
  int N, H;
  float c;  // scale * log2(e)
  float* sal;
  int* status;
  int adm_k;       // >= 1: fused admission with these arguments
  AdmitArgs adm;
};

__device__ __forceinline__ void cp_async16(uint32_t dst, const void* src) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() {
  asm volatile("cp.async.wait_all;" ::: "memory");
}

// Gather sampled query rows [ch*128, ch*128+128) of head h, chunks g0..g1-1,
// into swizzled K-major tiles (16-byte chunk c of row r at chunk c ^ (r % 8)).
// The index loads of all chunks are issued first, then the copies that
// depend on them; tok[c] keeps each thread's row (-1 past nq: a zero row).
__device__ __forceinline__ void gather_rows(const Params& p, int h, int g0, int g1, Smem& sm, int tid,
                                            int (&tok)[QS]) {
#pragma unroll
  for (int c = 0; c < QS; ++c) {
    const int i = (g0 + c) * BT + tid;
    tok[c] = (g0 + c < g1 && i < p.nq) ? __ldg(p.qidx + i) : -1;
    if (!dev_check(tok[c] < p.N, p.status)) tok[c] = -1;
  }
#pragma unroll
  for (int c = 0; c < QS; ++c) {
    const int ch = g0 + c;
    if (ch >= g1) break;
    uint8_t* tile = sm.qs[ch % QS];
    const uint32_t base = smem_addr(tile) + tid * 128;
    if (tok[c] >= 0) {
      const uint4* src = reinterpret_cast<const uint4*>(p.Q + ((size_t)tok[c] * p.H + h) * HD);
#pragma unroll
      for (int q = 0; q < 8; ++q) cp_async16(base + ((q ^ (tid & 7)) * 16), src + q);
    } else {
#pragma unroll
      for (int q = 0; q < 8; ++q)
        *reinterpret_cast<uint4*>(tile + tid * 128 + q * 16) = make_uint4(0, 0, 0, 0);
    }
  }
}

// The LSE of the gathered rows, in log2 units, into lse2 (+inf for zero rows,
// so they contribute exp2(-inf) = 0).
__device__ __forceinline__ void gather_lse(const Params& p, int h, int g0, int g1, Smem& sm, int tid,
                                           const int (&tok)[QS]) {
  float lv[QS];
#pragma unroll
  for (int c = 0; c < QS; ++c) lv[c] = tok[c] >= 0 ? p.lse[(size_t)h * p.N + tok[c]] : 0.f;
#pragma unroll
  for (int c = 0; c < QS; ++c)
    if (g0 + c < g1) sm.lse2[(g0 + c) % QS][tid] = tok[c] >= 0 ? lv[c] * 1.4426950408889634f : INFINITY;
}

// SHARED: the fused admission without head-specific retention (its own
// instantiation, so the per-head kernel's code is unchanged by it).
template <bool SHARED>
__global__ void __launch_bounds__(THREADS) saliency_kernel(const __grid_constant__ CUtensorMap tmK,
                                                           const Params p) {
  extern __shared__ uint8_t smem_raw[];
  const uintptr_t raw = reinterpret_cast<uintptr_t>(smem_raw);
  Smem& sm = *reinterpret_cast<Smem*>((raw + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5;
  const int nkt = (p.N + BT - 1) / BT;
  const int h = blockIdx.x / nkt, kt = blockIdx.x - h * nkt;
  const int nchunks = (p.nq + BT - 1) / BT;
  volatile int* abort_flag = &sm.abort_flag;
  volatile int* never = &sm.never;
  const uint32_t b_k = smem_addr(&sm.k_full), b_fin = smem_addr(&sm.fin_bar);
  const uint32_t b_mma[2] = {smem_addr(&sm.mma_bar[0]), smem_addr(&sm.mma_bar[1])};
  const bool issuer = (tid == 0);

  if (issuer) {
    sm.abort_flag = 0;
    sm.never = 0;
    mbar_init(b_k, 1);
    mbar_init(b_mma[0], 1);
    mbar_init(b_mma[1], 1);
    mbar_init(b_fin, 1);
    fence_barrier_init();
    mbar_arrive_expect_tx(b_k, TILE_BYTES);
    tma_load_3d(smem_addr(sm.k), &tmK, b_k, 0, h, kt * BT);
  }
  if (warp == 0) {
    tmem_alloc(smem_addr(&sm.tmem_base), TMEM_COLS);
    tmem_relinquish();
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
  bool k_ok = true;
  float acc = 0.f;
  uint32_t ph[2] = {0u, 0u};
  int issued = 0;  // MMAs issued (chunk index of the next one)
  auto issue = [&](int ch) {  // issuer only: Z^T of chunk ch into buffer ch % 2
    const uint32_t qaddr = smem_addr(sm.qs[ch % QS]);
#pragma unroll
    for (int kk = 0; kk < HD / 16; ++kk)
      mma_ss(tmem + (ch & 1) * 128, sdesc_sw128(smem_addr(sm.k) + kk * 32),
             sdesc_sw128(qaddr + kk * 32), IDESC, kk > 0);
    mma_commit(b_mma[ch & 1]);
  };
  bool stop = false;
  // The key tile (issued above) and the sampled rows come from the frame's
  // inputs, which precede the attention kernel: they are loaded while that
  // kernel finishes.  The LSE it writes is read after the wait.
  int tok[QS];
  gather_rows(p, h, 0, min(nchunks, QS), sm, tid, tok);
  grid_dep_wait();
  grid_dep_launch();
  for (int g0 = 0; g0 < nchunks && !stop; g0 += QS) {
    const int g1 = min(nchunks, g0 + QS);
    // every MMA that read the chunk buffers has completed (waited below)
    if (g0 > 0) gather_rows(p, h, g0, g1, sm, tid, tok);
    gather_lse(p, h, g0, g1, sm, tid, tok);
    cp_async_wait_all();
    fence_proxy_async_smem();
    tc_fence_before();
    __syncthreads();
    if (issuer) {
      tc_fence_after();
      if (g0 == 0) k_ok = mbar_wait(b_k, 0, abort_flag, WAIT_NS);
      for (; issued < min(g1, g0 + 2); ++issued) {
        if (k_ok) issue(issued);
        else mma_commit(b_mma[issued & 1]);
      }
    }
    for (int ch = g0; ch < g1; ++ch) {
      const int tb = ch & 1;
      const bool ok = mbar_wait(b_mma[tb], ph[tb], abort_flag, WAIT_NS);
      ph[tb] ^= 1;
      tc_fence_after();
      uint32_t z[128];
      if (ok) tmem_ld128(tmem + lane_off + tb * 128, z);
      tc_fence_before();
      // every thread has read Z^T(ch): its buffer can take chunk ch+2
      if (__syncthreads_or(!ok || *abort_flag)) {
        stop = true;
        break;
      }
      if (issuer && issued < g1) {
        tc_fence_after();
        if (k_ok) issue(issued);
        else mma_commit(b_mma[issued & 1]);
        ++issued;
      }
      const float* l2 = sm.lse2[ch % QS];
      float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
      for (int i = 0; i < 128; ++i) a4[i & 3] += ex2(fmaf(__uint_as_float(z[i]), p.c, -l2[i]));
      acc += (a4[0] + a4[1]) + (a4[2] + a4[3]);
    }
    __syncthreads();  // lse2 and the chunk buffers are refilled by the next group
  }
  const int j = kt * BT + tid;
  if (j < p.N && !*abort_flag) p.sal[(size_t)h * p.N + j] = acc;
  if (issuer) {
    mma_commit(b_fin);
    mbar_wait(b_fin, 0, never, DRAIN_NS);
    if (!k_ok || nchunks == 0) mbar_wait(b_k, 0, never, DRAIN_NS);
  }
  cp_async_wait_all();
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(p.status, kStatusTimeout);
  if (p.adm_k < 1) return;
  const bool cand = j < p.N && j >= p.adm.cand_lo;
  uint64_t* lists = reinterpret_cast<uint64_t*>(&sm.qs[0][0]);  // THREADS values
  if constexpr (SHARED) {
    // ---- fused admission without head-specific retention (Table 4): the
    // last head to finish a key tile ranks the tile's tokens by their
    // saliency summed over the heads (heads added in ascending order, as the
    // separate selection sums them); the last tile to finish merges the
    // tiles' lists, and every head's bank receives the same k rows
    __threadfence();  // this head's saliency before the tile's count
    __syncthreads();
    if (tid == 0) sm.last = atomicAdd(p.adm.done + kt, 1) == p.H - 1;
    __syncthreads();
    if (!sm.last) return;
    __threadfence();
    float sum = 0.f;
    if (cand)
      for (int hh = 0; hh < p.H; ++hh) sum += __ldcg(p.sal + (size_t)hh * p.N + j);
    sel::block_top_list<THREADS>(cand ? sel::pack_candidate(sum, j) : 0ull, lists,
                                 p.adm.lists + (size_t)kt * sel::kListK);
    __threadfence();  // the list before the count
    __syncthreads();
    if (tid == 0) {
      p.adm.done[kt] = 0;  // every head of this tile has counted
      sm.last = atomicAdd(p.adm.done + nkt, 1) == nkt - 1;
    }
    __syncthreads();
    if (!sm.last) return;
    __threadfence();
    int* ord = reinterpret_cast<int*>(&sm.qs[1][0]);
    sel::merge_head_lists<THREADS>(p.adm.lists, nkt, p.adm_k, p.adm.cand_lo, lists, ord);
    // every head's rows of the k tokens: 16-byte pieces (head, K or V, row,
    // piece), eight loads in flight per thread before their stores
    const int per_head = p.adm_k * 16, total = p.H * per_head;
    for (int w0 = tid; w0 < total; w0 += THREADS * 8) {
      uint4 v[8];
      uint4* dst[8];
#pragma unroll
      for (int u = 0; u < 8; ++u) {
        const int w = w0 + u * THREADS;
        dst[u] = nullptr;
        if (w >= total) continue;
        const int hh = w / per_head, rem = w - hh * per_head;
        const int which = rem / (p.adm_k * 8), r = (rem >> 3) % p.adm_k, c = rem & 7;
        const int tok = p.adm.cand_lo + ord[r];
        if (!dev_check(tok >= p.adm.cand_lo && tok < p.N && p.adm.M + r < p.adm.cap, p.status)) continue;
        const __nv_bfloat16* src = (which ? p.adm.V : p.adm.K) + ((size_t)tok * p.H + hh) * HD;
        dst[u] = reinterpret_cast<uint4*>((which ? p.adm.bankV : p.adm.bankK) +
                                          ((size_t)hh * p.adm.cap + p.adm.M + r) * HD) + c;
        v[u] = reinterpret_cast<const uint4*>(src)[c];
      }
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (dst[u]) *dst[u] = v[u];
    }
    if (p.adm.idx_out)
      for (int r = tid; r < p.adm_k; r += THREADS) p.adm.idx_out[r] = p.adm.cand_lo + ord[r];
    if (tid == 0) p.adm.done[nkt] = 0;
    return;
  }
  // ---- fused admission: this tile's best candidates, then the head's last
  // block merges the tiles' lists and appends
  sel::block_top_list<THREADS>(cand ? sel::pack_candidate(acc, j) : 0ull, lists,
                               p.adm.lists + ((size_t)h * nkt + kt) * sel::kListK);
  __threadfence();  // the list before the count
  __syncthreads();
  if (tid == 0) sm.last = atomicAdd(p.adm.done + h, 1) == nkt - 1;
  __syncthreads();
  if (!sm.last) return;
  __threadfence();
  int* ord = reinterpret_cast<int*>(&sm.qs[1][0]);
  sel::merge_head_lists<THREADS>(p.adm.lists + (size_t)h * nkt * sel::kListK, nkt, p.adm_k,
                                 p.adm.cand_lo, lists, ord);
  sel::append_rows<THREADS>(p.adm, h, ord);
  if (tid == 0) p.adm.done[h] = 0;  // every block of the head has counted
}

}  // namespace

cudaError_t saliency_setup() {
  const cudaError_t e = cudaFuncSetAttribute(saliency_kernel<false>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)SMEM_BYTES);
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(saliency_kernel<true>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)SMEM_BYTES);
}

cudaError_t launch_saliency(const SalArgs& a, cudaStream_t s) {
  if (a.nq > MAX_CHUNKS * BT) return cudaErrorInvalidValue;
  Params p;
  p.Q = a.Q;
  p.qidx = a.qidx;
  p.nq = a.nq;
  p.lse = a.lse;
  p.N = a.N;
  p.H = a.H;
  p.c = a.scale * 1.4426950408889634f;
  p.sal = a.sal;
  p.status = a.status;
  p.adm_k = 0;
  if (a.adm) {
    const int nc = a.N - a.adm->cand_lo;
    if (a.adm->sal != a.sal || !a.adm->lists || !a.adm->done || nc < 1 || a.adm->k < 1 ||
        a.adm->k > nc || a.adm->k > sel::kListK)
      return cudaErrorInvalidValue;
    p.adm = *a.adm;
    p.adm_k = a.adm->k;
  }
  const int nkt = (a.N + BT - 1) / BT;
  if (p.adm_k >= 1 && p.adm.shared)
    return launch_pdl(saliency_kernel<true>, dim3(a.H * nkt), dim3(THREADS), SMEM_BYTES, s, *a.tmK, p);
  return launch_pdl(saliency_kernel<false>, dim3(a.H * nkt), dim3(THREADS), SMEM_BYTES, s, *a.tmK, p);
}

}  // namespace regmem_dev
