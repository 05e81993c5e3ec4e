// Admission into the regulated memory.
//
// admit_kernel (Eq. 6, per head as in Sec. 3.3 "Head-Specific Token
// Retention"): one CTA per head selects the k candidates with the largest
// saliency -- order (saliency descending, token index ascending), so ties go
// to the lower index -- and appends their K and V rows, in ascending token
// order, after the M rows already in that head's bank.
// Selection is exact: the k-th largest saliency value T is found by a radix
// select over the order-preserving 32-bit pattern of the fp32 saliency (four
// passes of 8-bit digits, a shared-memory histogram per pass); every
// candidate above T is admitted, and of those equal to T the lowest token
// indices fill the remaining slots (a block scan in token order).  A second
// block scan over the admitted flags gives each admitted token its slot in
// ascending token order.  Rows are copied with 16-byte vector loads/stores
// (a 128-byte row is 8 lanes' worth).
//
// anchor_kernel (Eq. 4): the first frame's K and V rows of every head become
// the bank's first N rows.

#include "kernels.h"

namespace regmem_dev {

namespace {

constexpr int THREADS = 256;
constexpr int WARPS = THREADS / 32;
constexpr int PER = kMaxCandidates / THREADS;  // candidates per thread, at most
constexpr int HD = kHeadDim;

__device__ __forceinline__ uint32_t order_bits(float f) {
  const uint32_t u = __float_as_uint(f);
  return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive prefix sum over the block of one value per thread; returns this
// thread's offset.
__device__ __forceinline__ int block_exclusive_scan(int v, int* warp_sums) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const int y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[warp] = x;
  __syncthreads();
  if (warp == 0) {
    int w = lane < WARPS ? warp_sums[lane] : 0;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const int y = __shfl_up_sync(0xffffffffu, w, o);
      if (lane >= o) w += y;
    }
    if (lane < WARPS) warp_sums[lane] = w;  // inclusive prefix of warp totals
  }
  __syncthreads();
  const int base = warp ? warp_sums[warp - 1] : 0;
  __syncthreads();  // warp_sums may be reused by the next scan
  return base + x - v;
}

__global__ void __launch_bounds__(THREADS) admit_kernel(AdmitArgs a) {
  __shared__ int hist[256];
  __shared__ int warp_sums[WARPS];
  __shared__ int s_bin, s_above;
  extern __shared__ int ord[];  // [k] admitted token indices, ascending
  const int h = blockIdx.x, tid = threadIdx.x, lane = tid & 31;
  const int nc = a.N - a.cand_lo;
  const int per = (nc + THREADS - 1) / THREADS;  // contiguous candidates per thread
  const int first = tid * per;
  const int cnt = max(0, min(per, nc - first));
  const float* s = a.sal + (size_t)h * a.N + a.cand_lo;
  uint32_t key[PER];
#pragma unroll
  for (int i = 0; i < PER; ++i) key[i] = i < cnt ? order_bits(s[first + i]) : 0u;

  // ---- radix select of the k-th largest key
  uint32_t prefix = 0, mask = 0;
  int krem = a.k;
#pragma unroll 1
  for (int shift = 24; shift >= 0; shift -= 8) {
    hist[tid] = 0;  // THREADS == 256 bins
    __syncthreads();
#pragma unroll
    for (int i = 0; i < PER; ++i)
      if (i < cnt && (key[i] & mask) == prefix) atomicAdd(&hist[(key[i] >> shift) & 255u], 1);
    __syncthreads();
    if (tid < 32) {
      // lane l owns bins 8l..8l+7; find the bin b where the count of keys in
      // bins >= b first reaches krem
      int loc[8], lsum = 0;
#pragma unroll
      for (int q = 0; q < 8; ++q) {
        loc[q] = hist[lane * 8 + q];
        lsum += loc[q];
      }
      int suf = lsum;  // inclusive suffix sum over lanes >= lane
#pragma unroll
      for (int o = 1; o < 32; o <<= 1) {
        const int y = __shfl_down_sync(0xffffffffu, suf, o);
        if (lane + o < 32) suf += y;
      }
      int run = suf - lsum;  // keys in bins owned by higher lanes
#pragma unroll
      for (int q = 7; q >= 0; --q) {
        if (run < krem && run + loc[q] >= krem) {
          s_bin = lane * 8 + q;
          s_above = run;
        }
        run += loc[q];
      }
    }
    __syncthreads();
    krem -= s_above;
    prefix |= (uint32_t)s_bin << shift;
    mask |= 255u << shift;
    __syncthreads();  // s_bin / s_above are rewritten by the next pass
  }
  const uint32_t T = prefix;  // the k-th largest key; krem of the keys == T are admitted

  // ---- admitted flags in token order: all keys > T, and the first krem keys == T
  int n_eq = 0;
#pragma unroll
  for (int i = 0; i < PER; ++i) n_eq += (i < cnt && key[i] == T);
  int eq_rank = block_exclusive_scan(n_eq, warp_sums);
  uint32_t sel_bits = 0;
  int n_sel = 0;
#pragma unroll
  for (int i = 0; i < PER; ++i) {
    bool sel = false;
    if (i < cnt) {
      if (key[i] > T) sel = true;
      else if (key[i] == T) sel = (eq_rank++ < krem);
    }
    if (sel) {
      sel_bits |= 1u << i;
      ++n_sel;
    }
  }
  int slot = block_exclusive_scan(n_sel, warp_sums);
#pragma unroll
  for (int i = 0; i < PER; ++i)
    if (sel_bits & (1u << i)) ord[slot++] = a.cand_lo + first + i;
  __syncthreads();

  if (a.idx_out)
    for (int r = tid; r < a.k; r += THREADS) a.idx_out[(size_t)h * a.k + r] = ord[r];
  // ---- append: 8 x 16-byte chunks per 128-byte row, K then V
  const int work = a.k * 8 * 2;
  for (int w = tid; w < work; w += THREADS) {
    const int which = w / (a.k * 8);
    const int rem = w - which * a.k * 8;
    const int r = rem >> 3, c = rem & 7;
    const __nv_bfloat16* src = (which ? a.V : a.K) + ((size_t)ord[r] * a.H + h) * HD;
    __nv_bfloat16* dst = (which ? a.bankV : a.bankK) + ((size_t)h * a.cap + a.M + r) * HD;
    reinterpret_cast<uint4*>(dst)[c] = reinterpret_cast<const uint4*>(src)[c];
  }
  (void)lane;
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
                              (int)(kMaxCandidates * sizeof(int)));
}

cudaError_t launch_admit(const AdmitArgs& a, cudaStream_t s) {
  const int nc = a.N - a.cand_lo;
  if (nc < 1 || nc > kMaxCandidates || a.k < 0 || a.k > nc) return cudaErrorInvalidValue;
  if (a.k == 0) return cudaSuccess;
  admit_kernel<<<a.H, THREADS, (size_t)a.k * sizeof(int), s>>>(a);
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
