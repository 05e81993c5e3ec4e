// Admission into the regulated memory.
//
// Admission kernels (Eq. 6, per head as in Sec. 3.3 "Head-Specific Token
// Retention"); both append the admitted K and V rows, in ascending token
// order, after the M rows already in the head's bank.
// admit_lists_kernel (k <= 32): one block per (head, 128-key tile) keeps the
//   tile's best candidates; the head's last block merges the lists (the same
//   distributed selection the fused saliency kernel runs).
// admit_kernel (any k): one block per head runs the radix selection of
//   select.cuh over all of the head's candidates.
//
// anchor_kernel (Eq. 4): the first frame's K and V rows of every head become
// the bank's first N rows.

#include "kernels.h"
#include "ptx.cuh"
#include "select.cuh"

namespace regmem_dev {
using ptx::grid_dep_wait;
using ptx::grid_dep_launch;

namespace {

constexpr int THREADS = 256;
constexpr int WARPS = THREADS / 32;
constexpr int HD = kHeadDim;

__global__ void __launch_bounds__(THREADS) admit_kernel(AdmitArgs a) {
  __shared__ int red[sel::red_words<THREADS>()], ws[WARPS], bc[2];
  extern __shared__ uint32_t dyn[];  // keys [n], then the admitted positions [k]
  grid_dep_wait();  // the saliency kernel has finished
  grid_dep_launch();
  const int h = blockIdx.x;
  const int n = a.N - a.cand_lo;
  uint32_t* keys = dyn;
  int* ord = reinterpret_cast<int*>(dyn + n);
  sel::load_keys<THREADS>(a.sal + (size_t)h * a.N + a.cand_lo, n, keys);
  sel::select_topk<THREADS>(keys, n, a.k, ord, red, ws, bc);
  sel::append_rows<THREADS>(a, h, ord);
}

constexpr int LT = kTile;  // threads of the list kernel: one per key of the tile

__global__ void __launch_bounds__(LT) admit_lists_kernel(AdmitArgs a, int nkt) {
  __shared__ uint64_t lists[LT];
  __shared__ int ord[sel::kListK];
  __shared__ int last;
  grid_dep_wait();  // the saliency kernel has finished
  grid_dep_launch();
  const int h = blockIdx.x / nkt, kt = blockIdx.x - h * nkt, tid = threadIdx.x;
  const int j = kt * LT + tid;
  const bool cand = j < a.N && j >= a.cand_lo;
  const float s = cand ? a.sal[(size_t)h * a.N + j] : 0.f;
  sel::block_top_list<LT>(cand ? sel::pack_candidate(s, j) : 0ull, lists,
                          a.lists + ((size_t)h * nkt + kt) * sel::kListK);
  __threadfence();  // the list before the count
  __syncthreads();
  if (tid == 0) last = atomicAdd(a.done + h, 1) == nkt - 1;
  __syncthreads();
  if (!last) return;
  __threadfence();
  sel::merge_head_lists<LT>(a.lists + (size_t)h * nkt * sel::kListK, nkt, a.k, a.cand_lo, lists, ord);
  sel::append_rows<LT>(a, h, ord);
  if (tid == 0) a.done[h] = 0;
}

__global__ void anchor_kernel(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                              __nv_bfloat16* bankV, long long cap, int N, int H) {
  grid_dep_wait();
  grid_dep_launch();
  const long long total = (long long)N * H * 8;  // 16-byte chunks per tensor
  for (long long w = blockIdx.x * (long long)blockDim.x + threadIdx.x; w < 2 * total;
       w += (long long)gridDim.x * blockDim.x) {
    const int which = w >= total;
    const long long e = which ? w - total : w;
    const int c = (int)(e & 7);
    const long long nh = e >> 3;  // n * H + h
    const int h = (int)(nh % H);
    const long long n = nh / H;
    const uint4* src = reinterpret_cast<const uint4*>((which ? V : K) + nh * HD);
    uint4* dst = reinterpret_cast<uint4*>((which ? bankV : bankK) + ((size_t)h * cap + n) * HD);
    dst[c] = src[c];
  }
}

}  // namespace

cudaError_t admit_setup() {
  return cudaFuncSetAttribute(admit_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)(2 * kMaxCandidates * sizeof(int)));
}

cudaError_t launch_admit(const AdmitArgs& a, cudaStream_t s) {
  const int nc = a.N - a.cand_lo;
  if (nc < 1 || nc > kMaxCandidates || a.k < 0 || a.k > nc) return cudaErrorInvalidValue;
  if (a.k == 0) return cudaSuccess;
  if (a.k <= sel::kListK && a.lists && a.done) {
    const int nkt = (a.N + LT - 1) / LT;
    return launch_pdl(admit_lists_kernel, dim3(a.H * nkt), dim3(LT), 0, s, a, nkt);
  }
  return launch_pdl(admit_kernel, dim3(a.H), dim3(THREADS), (size_t)(nc + a.k) * sizeof(int), s, a);
}

cudaError_t launch_anchor(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                          __nv_bfloat16* bankV, long long cap, int N, int H, cudaStream_t s) {
  const long long work = 2LL * N * H * 8;
  int blocks = (int)((work + 255) / 256);
  if (blocks > 4096) blocks = 4096;
  return launch_pdl(anchor_kernel, dim3(blocks), dim3(256), 0, s, K, V, bankK, bankV, cap, N, H);
}

}  // namespace regmem_dev
