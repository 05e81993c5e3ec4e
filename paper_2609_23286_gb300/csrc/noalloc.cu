// Allocation-free variant of the attend step (regmem_attend_frame_noalloc).
//
// Some callers cannot allocate device memory at the point where they run the
// attention: code that executes inside another framework's memory pool or
// arena, plugins that are handed pre-sized buffers, and real-time loops where
// an allocation could block on the driver.  For them this entry point runs
// the same attention kernel (with its split-piece merge) and the same
// LSE-saliency kernel as regmem_attend_frame, but on caller-owned tensors
// only: no handle, no cudaMalloc/cudaFree, no allocating library call.  The
// kernels' scratch -- the split partials, the LSE rows and the sampled-query
// list -- lives in one file-scope device array of fixed size, which every GPU
// that loads this library holds until the process exits.

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <cmath>
#include <mutex>

#include "kernels.h"
#include "regmem.h"

namespace regmem_dev {
namespace {

constexpr int kMaxCtas = 160;               // split partials for one CTA on each of up to 160 SMs
constexpr size_t kMaxLse = 262144;          // heads * tokens per frame
constexpr int kMaxSampled = 8192;           // sampled queries per frame

struct NoAllocScratch {
  __nv_bfloat16 part_o[(size_t)kMaxCtas * 2 * kUnitRows * kHeadDim];  // first / last piece of each CTA
  float part_lse[(size_t)kMaxCtas * 2 * kUnitRows];
  float lse[kMaxLse];
  int qidx[kMaxSampled];
};

// 11.9 MB; shared by every call on a device.
static __device__ __align__(256) NoAllocScratch g_scratch;

constexpr int kMaxDevices = 64;
struct DeviceSetup {
  bool done = false;
  NoAllocScratch* scratch = nullptr;  // device address of g_scratch on this device
  int sms = 0;
  int ctas_per_sm = 0;
};
DeviceSetup g_setup[kMaxDevices];
std::mutex g_setup_mutex;

// Writes the sampled query tokens: top-left query of each ds x ds window of
// the patch grid, row-major (Sec. 3.3, Head-Specific Token Retention).
__global__ void sampled_tokens_kernel(int* qidx, int nq, int n_special, int grid_w, int ds,
                                      int cols) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < nq) qidx[i] = n_special + (i / cols) * ds * grid_w + (i % cols) * ds;
}

PFN_cuTensorMapEncodeTiled_v12000 encoder() {
  static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
  });
  return fn;
}

// 3-D view (channel, d1, d2) of a bf16 tensor with 128-byte rows; box 64 x b1 x b2.
bool encode3d(CUtensorMap* m, const void* ptr, uint64_t d1, uint64_t d2, uint64_t s1, uint64_t s2,
              uint32_t b1, uint32_t b2) {
  auto enc = encoder();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, d1, d2};
  cuuint64_t strides[2] = {s1, s2};
  cuuint32_t box[3] = {(cuuint32_t)kHeadDim, b1, b2};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

}  // namespace
}  // namespace regmem_dev

using namespace regmem_dev;

extern "C" REGMEM_API regmem_status regmem_attend_frame_noalloc(const regmem_frame_desc* fd, int32_t heads,
                                                     const void* Q, const void* K, const void* V,
                                                     const void* bankK, const void* bankV,
                                                     int64_t bank_rows, int64_t M, void* out,
                                                     float* saliency, int32_t* status,
                                                     void* stream_) {
  cudaStream_t stream = static_cast<cudaStream_t>(stream_);
  // status is required: with no handle there is no later call that could
  // report an expired device-side wait, so the caller's word is the only
  // place the kernels can record it
  if (!fd || heads < 1 || !Q || !K || !V || !out || !saliency || !status) return REGMEM_ERR_ARG;
  const int ds = fd->ds == 0 ? 2 : fd->ds;
  if (fd->n_special < 0 || fd->grid_h < 1 || fd->grid_w < 1 || ds < 1 ||
      fd->n_tokens != fd->n_special + fd->grid_h * fd->grid_w || fd->scale < 0.f ||
      !std::isfinite(fd->scale))
    return REGMEM_ERR_ARG;
  if (M < 0 || (M > 0 && (!bankK || !bankV || bank_rows < M)) || M > (1LL << 31) - 1)
    return REGMEM_ERR_ARG;
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(out) || !aligned16(saliency) ||
      (M > 0 && (!aligned16(bankK) || !aligned16(bankV))) ||
      (reinterpret_cast<uintptr_t>(status) & 3u))
    return REGMEM_ERR_ARG;
  const int N = fd->n_tokens;
  const int cols = (fd->grid_w + ds - 1) / ds;
  const int nq = ((fd->grid_h + ds - 1) / ds) * cols;
  // sizes beyond what the static scratch holds
  if (N > 65536 || (size_t)heads * N > kMaxLse || nq > kMaxSampled) return REGMEM_ERR_UNSUPPORTED;

  int dev = 0;
  if (cudaGetDevice(&dev) != cudaSuccess) return REGMEM_ERR_CUDA;
  if (dev < 0 || dev >= kMaxDevices) return REGMEM_ERR_UNSUPPORTED;
  DeviceSetup setup;
  {
    // Once per device, with that device current: the device address of the
    // scratch array (its host-side name is only a stand-in, never passed to a
    // kernel), the SM count and the kernels' attributes.
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    DeviceSetup& s = g_setup[dev];
    if (!s.done) {
      void* ptr = nullptr;
      if (cudaGetSymbolAddress(&ptr, g_scratch) != cudaSuccess || !ptr) return REGMEM_ERR_CUDA;
      if (cudaDeviceGetAttribute(&s.sms, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess)
        return REGMEM_ERR_CUDA;
      if (attn_setup() != cudaSuccess || saliency_setup() != cudaSuccess) return REGMEM_ERR_CUDA;
      s.ctas_per_sm = attn_ctas_per_sm();
      s.scratch = static_cast<NoAllocScratch*>(ptr);
      s.done = true;
    }
    setup = s;
  }
  NoAllocScratch* sc = setup.scratch;

  const AttnPlan pl = attn_plan(N, heads, (int)M);
  long long G = (long long)setup.sms * setup.ctas_per_sm;
  if (G > pl.total) G = pl.total;
  if (G > kMaxCtas) return REGMEM_ERR_UNSUPPORTED;  // more CTAs than the partial scratch holds

  CUtensorMap tq, tk, tv, tbk, tbv;
  const uint64_t rowb = kHeadDim * 2;
  if (!encode3d(&tq, Q, heads, N, rowb, rowb * heads, 1, kTile) ||
      !encode3d(&tk, K, heads, N, rowb, rowb * heads, 1, kTile) ||
      !encode3d(&tv, V, heads, N, rowb, rowb * heads, 1, kTile))
    return REGMEM_ERR_CUDA;
  if (M > 0) {
    if (!encode3d(&tbk, bankK, bank_rows, heads, rowb, rowb * bank_rows, kTile, 1) ||
        !encode3d(&tbv, bankV, bank_rows, heads, rowb, rowb * bank_rows, kTile, 1))
      return REGMEM_ERR_CUDA;
  } else {  // no bank tiles are read when M == 0
    tbk = tk;
    tbv = tv;
  }

  int* st = status;
  sampled_tokens_kernel<<<(nq + 255) / 256, 256, 0, stream>>>(sc->qidx, nq, fd->n_special,
                                                               fd->grid_w, ds, cols);
  if (cudaGetLastError() != cudaSuccess) return REGMEM_ERR_CUDA;

  const float scale = fd->scale == 0.f ? 1.f / std::sqrt((float)kHeadDim) : fd->scale;
  AttnArgs a = {};
  a.tmQ = &tq;
  a.tmK = &tk;
  a.tmV = &tv;
  a.tmBK = &tbk;
  a.tmBV = &tbv;
  a.N = N;
  a.H = heads;
  a.M = (int)M;
  a.scale = scale;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.lse = sc->lse;
  a.part_o = sc->part_o;
  a.part_lse = sc->part_lse;
  a.max_phases = 1;  // the fixed scratch holds two partial slots per CTA
  a.status = st;
  a.wait_ns = 2000000000ull;  // 2 s
  a.fault_skip_kv = -1;
  a.grid = (int)G;
  if (launch_attention(a, stream) != cudaSuccess) return REGMEM_ERR_CUDA;

  SalArgs sa = {};
  sa.tmK = &tk;
  sa.Q = static_cast<const __nv_bfloat16*>(Q);
  sa.qidx = sc->qidx;
  sa.nq = nq;
  sa.lse = sc->lse;
  sa.N = N;
  sa.H = heads;
  sa.scale = scale;
  sa.sal = saliency;
  sa.status = st;
  if (launch_saliency(sa, stream) != cudaSuccess) return REGMEM_ERR_CUDA;
  return REGMEM_OK;
}
