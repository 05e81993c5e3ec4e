// Admission into the regulated memory.
//
// admit_kernel (Eq. 6, per head as in Sec. 3.3 "Head-Specific Token
// Retention"): one CTA per head selects the k candidates with the largest
// saliency -- order (saliency descending, token index ascending), so ties go
// to the lower index -- and appends their K and V rows, in ascending token
// order, after the M rows already in that head's bank.  Selection is exact:
// each candidate becomes a unique 64-bit key (order-preserving bits of the
// fp32 saliency, then the complemented token index) and the keys are sorted
// with a bitonic network in shared memory.  Rows are copied with 16-byte
// vector loads/stores (a 128-byte row is 8 lanes' worth).
//
// anchor_kernel (Eq. 4): the first frame's K and V rows of every head become
// the bank's first N rows.

#include "kernels.h"

namespace regmem_dev {

namespace {

constexpr int THREADS = 1024;
constexpr int HD = kHeadDim;

__device__ __forceinline__ uint32_t order_bits(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

__global__ void __launch_bounds__(THREADS) admit_kernel(AdmitArgs a, int pow2) {
  extern __shared__ unsigned long long keys[];  // [pow2] sort keys, then sel[k], ord[k]
  int* sel = reinterpret_cast<int*>(keys + pow2);  // selected token indices (unordered)
  int* ord = sel + a.k;                            // same, ascending
  const int h = blockIdx.x, tid = threadIdx.x;
  const int nc = a.N - a.cand_lo;
  const float* s = a.sal + (size_t)h * a.N;
  for (int i = tid; i < pow2; i += THREADS) {
    unsigned long long key = 0ull;  // padding sorts last
    if (i < nc) {
      const int j = a.cand_lo + i;
      key = ((unsigned long long)order_bits(s[j]) << 32) | (unsigned long long)(0xFFFFFFFFu - (uint32_t)j);
    }
    keys[i] = key;
  }
  __syncthreads();
  // Bitonic sort, descending.
  for (int size = 2; size <= pow2; size <<= 1) {
    for (int stride = size >> 1; stride > 0; stride >>= 1) {
      for (int i = tid; i < (pow2 >> 1); i += THREADS) {
        const int lo = 2 * i - (i & (stride - 1));
        const int hi = lo + stride;
        const bool desc = (lo & size) == 0;
        const unsigned long long x = keys[lo], y = keys[hi];
        if ((x < y) == desc) {
          keys[lo] = y;
          keys[hi] = x;
        }
      }
      __syncthreads();
    }
  }
  for (int r = tid; r < a.k; r += THREADS)
    sel[r] = (int)(0xFFFFFFFFu - (uint32_t)(keys[r] & 0xFFFFFFFFull));
  __syncthreads();
  // Ascending token order: a token's slot is the number of chosen tokens below it.
  for (int r = tid; r < a.k; r += THREADS) {
    const int j = sel[r];
    int rank = 0;
    for (int q = 0; q < a.k; ++q) rank += (sel[q] < j);
    ord[rank] = j;
  }
  __syncthreads();
  if (a.idx_out)
    for (int r = tid; r < a.k; r += THREADS) a.idx_out[(size_t)h * a.k + r] = ord[r];
  // Append: 8 x 16-byte chunks per 128-byte row, K then V.
  const int work = a.k * 8 * 2;
  for (int w = tid; w < work; w += THREADS) {
    const int which = w / (a.k * 8);
    const int rem = w - which * a.k * 8;
    const int r = rem >> 3, c = rem & 7;
    const __nv_bfloat16* src = (which ? a.V : a.K) + ((size_t)ord[r] * a.H + h) * HD;
    __nv_bfloat16* dst = (which ? a.bankV : a.bankK) + ((size_t)h * a.cap + a.M + r) * HD;
    reinterpret_cast<uint4*>(dst)[c] = reinterpret_cast<const uint4*>(src)[c];
  }
}

__global__ void anchor_kernel(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                              __nv_bfloat16* bankV, long long cap, int N, int H) {
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
                              (int)(kMaxCandidates * (sizeof(unsigned long long) + 2 * sizeof(int))));
}

cudaError_t launch_admit(const AdmitArgs& a, cudaStream_t s) {
  const int nc = a.N - a.cand_lo;
  if (nc < 1 || nc > kMaxCandidates || a.k < 0 || a.k > nc) return cudaErrorInvalidValue;
  if (a.k == 0) return cudaSuccess;
  int pow2 = 2;
  while (pow2 < nc) pow2 <<= 1;
  const size_t smem = pow2 * sizeof(unsigned long long) + 2 * (size_t)a.k * sizeof(int);
  admit_kernel<<<a.H, THREADS, smem, s>>>(a, pow2);
  return cudaGetLastError();
}

cudaError_t launch_anchor(const __nv_bfloat16* K, const __nv_bfloat16* V, __nv_bfloat16* bankK,
                          __nv_bfloat16* bankV, long long cap, int N, int H, cudaStream_t s) {
  const long long work = 2LL * N * H * 8;
  int blocks = (int)((work + 255) / 256);
  if (blocks > 4096) blocks = 4096;
  anchor_kernel<<<blocks, 256, 0, s>>>(K, V, bankK, bankV, cap, N, H);
  return cudaGetLastError();
}

}  // namespace regmem_dev
