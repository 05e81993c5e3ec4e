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
// The key tile arrives by TMA; sampled query rows are gathered with 16-byte
// loads into a 128-byte-swizzled tile, two chunks double-buffered so the next
// chunk's MMA overlaps the current chunk's exponentials.

#include "kernels.h"
#include "ptx.cuh"

namespace regmem_dev {
using namespace ptx;

namespace {

constexpr int BT = kTile, HD = kHeadDim;
constexpr int TILE_BYTES = BT * HD * 2;
constexpr int THREADS = 128;
constexpr uint32_t TMEM_COLS = 256;  // two 128-column Z^T buffers
constexpr uint64_t WAIT_NS = 2000000000ull;
constexpr uint64_t DRAIN_NS = 200000000ull;
constexpr uint32_t IDESC = idesc_bf16_f32(128, 128, false, false);
constexpr int MAX_CHUNKS = 64;  // sampled queries <= 8192

struct Smem {
  uint8_t k[TILE_BYTES];
  uint8_t qs[2][TILE_BYTES];
  float lse2[2][BT];
  uint64_t k_full, mma_bar[2], fin_bar;
  uint32_t tmem_base;
  int abort_flag;
  int never;
};
// At least 80 KB so no more than two CTAs share an SM: two 256-column TMEM
// allocations fill the SM's 512 columns.
constexpr size_t SMEM_BYTES = (sizeof(Smem) + 1024 > 80 * 1024) ? sizeof(Smem) + 1024 : 80 * 1024;

struct Params {
  const __nv_bfloat16* Q;
  const int* qidx;
  int nq;
  const float* lse;
  int N, H;
  float c;  // scale * log2(e)
  float* sal;
  int* status;
};

// Gather sampled query rows [chunk*128, chunk*128+128) of head h into a
// swizzled K-major tile, and their LSE (in log2 units) into lse2.  Rows past
// nq are zero with lse2 = +inf, so they contribute exp2(-inf) = 0.
__device__ __forceinline__ void gather_chunk(const Params& p, int h, int chunk, uint8_t* tile,
                                             float* lse2, int tid) {
  const int i = chunk * BT + tid;  // one sampled row per thread
  uint4 v[8];
  float l2 = INFINITY;
  if (i < p.nq) {
    const int tok = p.qidx[i];
    const uint4* src = reinterpret_cast<const uint4*>(p.Q + ((size_t)tok * p.H + h) * HD);
#pragma unroll
    for (int c = 0; c < 8; ++c) v[c] = src[c];
    l2 = p.lse[(size_t)h * p.N + tok] * 1.4426950408889634f;
  } else {
#pragma unroll
    for (int c = 0; c < 8; ++c) v[c] = make_uint4(0, 0, 0, 0);
  }
#pragma unroll
  for (int c = 0; c < 8; ++c)
    *reinterpret_cast<uint4*>(tile + tid * 128 + ((c ^ (tid & 7)) * 16)) = v[c];
  lse2[tid] = l2;
}

__global__ void __launch_bounds__(THREADS) saliency_kernel(const __grid_constant__ CUtensorMap tmK,
                                                           const Params p) {
  extern __shared__ uint8_t smem_raw[];
  const uintptr_t raw = reinterpret_cast<uintptr_t>(smem_raw);
  Smem& sm = *reinterpret_cast<Smem*>((raw + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  const int nkt = (p.N + BT - 1) / BT;
  const int h = blockIdx.x / nkt, kt = blockIdx.x - h * nkt;
  const int nchunks = (p.nq + BT - 1) / BT;
  volatile int* abort_flag = &sm.abort_flag;
  volatile int* never = &sm.never;
  const uint32_t b_k = smem_addr(&sm.k_full), b_fin = smem_addr(&sm.fin_bar);
  const uint32_t b_mma[2] = {smem_addr(&sm.mma_bar[0]), smem_addr(&sm.mma_bar[1])};

  if (tid == 0) {
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
  if (nchunks > 0) gather_chunk(p, h, 0, sm.qs[0], sm.lse2[0], tid);
  fence_proxy_async_smem();
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;
  const uint32_t lane_off = (uint32_t)(warp * 32) << 16;
  const bool elected = (tid == 0);
  bool k_ok = true;
  if (elected) {
    k_ok = mbar_wait(b_k, 0, abort_flag, WAIT_NS);
    if (k_ok && nchunks > 0) {
#pragma unroll
      for (int kk = 0; kk < HD / 16; ++kk)
        mma_ss(tmem, sdesc_sw128(smem_addr(sm.k) + kk * 32), sdesc_sw128(smem_addr(sm.qs[0]) + kk * 32),
               IDESC, kk > 0);
    }
    mma_commit(b_mma[0]);
  }
  float acc = 0.f;
  uint32_t ph[2] = {0u, 0u};
  for (int ch = 0; ch < nchunks; ++ch) {
    const int buf = ch & 1;
    const bool ok = mbar_wait(b_mma[buf], ph[buf], abort_flag, WAIT_NS);
    ph[buf] ^= 1;
    tc_fence_before();
    // After this barrier every thread is done with chunk ch-1 (its Z^T load
    // and its lse2 reads) and the MMA of chunk ch-1 has completed, so the
    // other buffers can be refilled for chunk ch+1.
    if (__syncthreads_or(!ok || *abort_flag)) break;
    if (ch + 1 < nchunks) {
      gather_chunk(p, h, ch + 1, sm.qs[buf ^ 1], sm.lse2[buf ^ 1], tid);
      fence_proxy_async_smem();
    }
    tc_fence_before();
    __syncthreads();
    if (elected && ch + 1 < nchunks) {
      tc_fence_after();
      if (k_ok) {
#pragma unroll
        for (int kk = 0; kk < HD / 16; ++kk)
          mma_ss(tmem + (buf ^ 1) * 128, sdesc_sw128(smem_addr(sm.k) + kk * 32),
                 sdesc_sw128(smem_addr(sm.qs[buf ^ 1]) + kk * 32), IDESC, kk > 0);
      }
      mma_commit(b_mma[buf ^ 1]);
    }
    tc_fence_after();
    uint32_t z[128];
    tmem_ld128(tmem + lane_off + buf * 128, z);
    const float* l2 = sm.lse2[buf];
    float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
    for (int i = 0; i < 128; ++i) a4[i & 3] += ex2(fmaf(__uint_as_float(z[i]), p.c, -l2[i]));
    acc += (a4[0] + a4[1]) + (a4[2] + a4[3]);
  }
  const int j = kt * BT + tid;
  if (j < p.N && !*abort_flag) p.sal[(size_t)h * p.N + j] = acc;
  if (elected) {
    mma_commit(b_fin);
    mbar_wait(b_fin, 0, never, DRAIN_NS);
    if (!k_ok) mbar_wait(b_k, 0, never, DRAIN_NS);
  }
  tc_fence_before();
  __syncthreads();
  if (warp == 0) {
    tc_fence_after();
    tmem_dealloc(tmem, TMEM_COLS);
  }
  if (tid == 0 && sm.abort_flag) atomicOr(p.status, kStatusTimeout);
}

}  // namespace

cudaError_t saliency_setup() {
  return cudaFuncSetAttribute(saliency_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
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
  const int nkt = (a.N + BT - 1) / BT;
  saliency_kernel<<<a.H * nkt, THREADS, SMEM_BYTES, s>>>(*a.tmK, p);
  return cudaGetLastError();
}

}  // namespace regmem_dev
