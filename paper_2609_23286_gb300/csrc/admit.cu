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
// admit_shared_kernel (any k): the selection without head-specific
//   retention (the ablation of Sec. 4.5, Table 4): one index set for all heads,
//   ranked by the head sum of the saliency (equivalently its head mean).
//
// copy_rows_kernel: rows [lo, lo + n) of the frame appended after row M of
// every head's bank, in token order.  It serves the first frame (Eq. 4: all N
// rows become the anchor) and an admission of every candidate (k equal to
// their count, e.g. the unregulated full-KV stream).

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

// One block per head: the candidates' head-summed saliency (fp32, heads added
// in ascending order, so every block forms the same keys) is ranked as in
// admit_kernel, and the block appends the chosen rows of its own head.
__global__ void __launch_bounds__(THREADS) admit_shared_kernel(AdmitArgs a) {
  __shared__ int red[sel::red_words<THREADS>()], ws[WARPS], bc[2];
  extern __shared__ uint32_t dyn[];  // keys [n], then the admitted positions [k]
  grid_dep_wait();  // the saliency kernel has finished
  grid_dep_launch();
  const int h = blockIdx.x;
  const int n = a.N - a.cand_lo;
  uint32_t* keys = dyn;
  int* ord = reinterpret_cast<int*>(dyn + n);
  for (int i = threadIdx.x; i < n; i += THREADS) {
    float sum = 0.f;
    for (int hh = 0; hh < a.H; ++hh) sum += __ldcg(a.sal + (size_t)hh * a.N + a.cand_lo + i);
    keys[i] = sel::order_bits(sum);
  }
  __syncthreads();
  sel::select_topk<THREADS>(keys, n, a.k, ord, red, ws, bc);
  AdmitArgs b = a;
  b.idx_out = nullptr;  // one index list, written by block 0
  sel::append_rows<THREADS>(b, h, ord);
  if (h == 0 && a.idx_out)
    for (int r = threadIdx.x; r < a.k; r += THREADS) a.idx_out[r] = a.cand_lo + ord[r];
}

__global__ void copy_rows_kernel(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                                 __nv_bfloat16* bankV, long long cap, long long M, int lo, int n,
                                 int H, int32_t* idx_out, int idx_rows, int n_tokens, int* status) {
  grid_dep_wait();
  grid_dep_launch();
  const long long total = (long long)n * H * 8;  // 16-byte chunks per tensor
  for (long long w = blockIdx.x * (long long)blockDim.x + threadIdx.x; w < 2 * total;
       w += (long long)gridDim.x * blockDim.x) {
    const int which = w >= total;
    const long long e = which ? w - total : w;
    const int c = (int)(e & 7);
    const long long rh = e >> 3;  // r * H + h
    const int h = (int)(rh % H);
    const long long r = rh / H;
    if (!dev_check(lo + r < n_tokens && M + r < cap, status)) continue;
    const uint4* src = reinterpret_cast<const uint4*>((which ? V : K) + ((lo + r) * H + h) * HD);
    uint4* dst = reinterpret_cast<uint4*>((which ? bankV : bankK) + ((size_t)h * cap + M + r) * HD);
    dst[c] = src[c];
    if (idx_out && !which && c == 0 && h < idx_rows) idx_out[(size_t)h * n + r] = (int32_t)(lo + r);
  }
}

// idx_out (optional) receives lo + r for r < n, in `idx_rows` rows of n.
cudaError_t launch_copy_rows(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                             __nv_bfloat16* bankV, long long cap, long long M, int lo, int n, int H,
                             int32_t* idx_out, int idx_rows, int n_tokens, int* status,
                             cudaStream_t s) {
  const long long work = 2LL * n * H * 8;
  int blocks = (int)((work + 255) / 256);
  if (blocks > 4096) blocks = 4096;
  return launch_pdl(copy_rows_kernel, dim3(blocks), dim3(256), 0, s, K, V, bankK, bankV, cap, M, lo, n,
                    H, idx_out, idx_rows, n_tokens, status);
}

}  // namespace

cudaError_t admit_setup() {
  cudaError_t e = cudaFuncSetAttribute(admit_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       (int)(2 * kMaxCandidates * sizeof(int)));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(admit_shared_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              (int)(2 * kMaxCandidates * sizeof(int)));
}

cudaError_t launch_admit(const AdmitArgs& a, cudaStream_t s) {
  const int nc = a.N - a.cand_lo;
  if (nc < 1 || nc > kMaxCandidates || a.k < 0 || a.k > nc) return cudaErrorInvalidValue;
  if (a.k == 0) return cudaSuccess;
  if (a.k == nc)  // every candidate: nothing to rank
    return launch_copy_rows(a.K, a.V, a.bankK, a.bankV, a.cap, a.M, a.cand_lo, nc, a.H, a.idx_out, a.H,
                            a.N, a.status, s);
  if (a.k <= sel::kListK && a.lists && a.done) {
    const int nkt = (a.N + LT - 1) / LT;
    return launch_pdl(admit_lists_kernel, dim3(a.H * nkt), dim3(LT), 0, s, a, nkt);
  }
  return launch_pdl(admit_kernel, dim3(a.H), dim3(THREADS), (size_t)(nc + a.k) * sizeof(int), s, a);
}

cudaError_t launch_admit_shared(const AdmitArgs& a, cudaStream_t s) {
  const int nc = a.N - a.cand_lo;
  if (nc < 1 || nc > kMaxCandidates || a.k < 0 || a.k > nc) return cudaErrorInvalidValue;
  if (a.k == 0) return cudaSuccess;
  if (a.k == nc)  // every candidate; one index list
    return launch_copy_rows(a.K, a.V, a.bankK, a.bankV, a.cap, a.M, a.cand_lo, nc, a.H, a.idx_out, 1,
                            a.N, a.status, s);
  return launch_pdl(admit_shared_kernel, dim3(a.H), dim3(THREADS), (size_t)(nc + a.k) * sizeof(int), s, a);
}

cudaError_t launch_anchor(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                          __nv_bfloat16* bankV, long long cap, int N, int H, int* status,
                          cudaStream_t s) {
  return launch_copy_rows(K, V, bankK, bankV, cap, 0, 0, N, H, nullptr, 0, N, status, s);
}

}  // namespace regmem_dev
