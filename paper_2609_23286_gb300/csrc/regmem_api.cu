// C ABI of libregmem.so (declared in include/regmem.h): handle, argument and
// state validation, HBM bank ownership, TMA descriptor set-up and kernel
// launches.  Every compute step runs in this library's kernels.

#include <cuda.h>
#include <cudaTypedefs.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <mutex>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "kernels.h"
#include "regmem.h"

using namespace regmem_dev;

namespace {

// One NVTX range per exported call, in the "regmem" domain, so that a
// timeline (nsys, ncu's NVTX filters) shows which library call enqueued
// which kernels.  With no tool attached a push/pop is a call through a null
// function pointer check.
nvtxDomainHandle_t nvtx_domain() {
  static nvtxDomainHandle_t d = nvtxDomainCreateA("regmem");
  return d;
}
struct NvtxRange {
  explicit NvtxRange(const char* name) {
    nvtxEventAttributes_t a = {};
    a.version = NVTX_VERSION;
    a.size = NVTX_EVENT_ATTRIB_STRUCT_SIZE;
    a.messageType = NVTX_MESSAGE_TYPE_ASCII;
    a.message.ascii = name;
    nvtxDomainRangePushEx(nvtx_domain(), &a);
  }
  ~NvtxRange() { nvtxDomainRangePop(nvtx_domain()); }
  NvtxRange(const NvtxRange&) = delete;
  NvtxRange& operator=(const NvtxRange&) = delete;
};

}  // namespace

#define REGMEM_RANGE NvtxRange nvtx_range_(__func__)

struct regmem {
  int layers = 0, heads = 0, head_dim = 0, budget = 0;
  bool frame_set = false;
  int device = 0;
  int N = 0, n_special = 0, grid_h = 0, grid_w = 0, ds = 2, cand_lo = 0, nq = 0;
  int max_frames = 0;
  float scale = 0.f;
  long long cap = 0;
  cudaStream_t stream = nullptr;

  std::vector<long long> len;
  std::vector<int> pending;
  std::vector<const __nv_bfloat16*> pK, pV;
  std::vector<float*> pS;

  __nv_bfloat16* bankK = nullptr;  // [layers][H][cap][64]
  __nv_bfloat16* bankV = nullptr;
  std::vector<CUtensorMap> tmBK, tmBV;

  float* lse = nullptr;       // [layers][H][N]: each layer's attention writes its own rows
  int lse_layer = 0;          // layer of the last attention (regmem_copy_lse)
  int* qidx = nullptr;        // [nq]
  __nv_bfloat16* part_o = nullptr;  // split-KV partials
  float* part_lse = nullptr;
  int* head_done = nullptr;   // completion counters of the distributed selection (per head or per key tile)
  // the attention's launch clock: kClockSlots start words, then as many end
  // words, one pair per launch since regmem_profile_enable
  unsigned long long* kclock = nullptr;
  long long clk_next = 0;
  std::vector<unsigned char> clk_frame;  // per clocked launch: 1 = frame attention
  uint64_t* adm_lists = nullptr;  // per-(head, key tile) candidate lists, [H][nkt][32]
  int attn_grid = 0;
  int attn_ctas_per_sm = 0;
  int* status_host = nullptr; // mapped pinned word written by kernels
  int* status_dev = nullptr;
  // bounded waits of the attention kernel, and the one-shot fault of
  // regmem_debug_set (failure-detection tests)
  unsigned long long wait_ns = 2000000000ull;
  int fault_skip_kv = -1;

  // staging of the host-buffer entry points (allocated by regmem_set_frame)
  __nv_bfloat16* stQ = nullptr;
  __nv_bfloat16* stOut = nullptr;
  float* stSal = nullptr;
  std::vector<__nv_bfloat16*> stK, stV;
  // regmem_attend_admit_host: six staging sets used in turn, copies in and
  // out on streams of their own, so one call's copies overlap the
  // neighbouring calls' kernels.  A set's inputs are read until the call's
  // side work ends (with overlap, inside the next call's attention) and its
  // outputs are copied out after that, so a set is free again only a few
  // calls later: with two sets the input copies waited for it, and six ran
  // the host-buffer stream faster than three.
  static constexpr unsigned kHostSets = 6;
  struct HostSet {
    __nv_bfloat16 *q = nullptr, *k = nullptr, *v = nullptr, *out = nullptr;
    float* sal = nullptr;
    cudaEvent_t h2d = nullptr, done = nullptr, d2h = nullptr;  // inputs in, kernels done, outputs out
    bool used = false;
  } hs[kHostSets];
  unsigned hs_next = 0;
  cudaStream_t cstream = nullptr;  // host->device copies of the host-buffer path
  cudaStream_t dstream = nullptr;  // device->host copies

  // regmem_set_overlap: the saliency and admission of regmem_attend_admit run
  // on a side stream of the lowest priority, ordered after the call's
  // attention (event main_ev); the next attention of a layer whose side work
  // is still unwaited waits for all side work so far (event side_ev).
  bool overlap = false;
  cudaStream_t sstream = nullptr;
  cudaEvent_t main_ev = nullptr, side_ev = nullptr;
  long long side_seq = 0;      // side submissions so far (side_ev marks the last)
  long long covered_seq = 0;   // side submissions the handle's stream has waited for
  std::vector<long long> side_seq_of;  // per layer: its last side submission

  // measurement (regmem_profile_*)
  regmem_profile prof = {};
  int time_every = 0;          // time every n-th attention launch (0: none)
  long long attn_launch_no = 0;
  std::vector<cudaEvent_t> ev_ring;  // triples: [3i] before, [3i+1] after the attention, [3i+2] after the merge
  std::vector<int> ev_busy;
  size_t ev_next = 0;

  std::string err;
};

namespace {

regmem_status fail(regmem_t* h, regmem_status s, const char* fmt, ...) {
  if (h) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof(buf), fmt, ap);
    va_end(ap);
    h->err = buf;
  }
  return s;
}

regmem_status cuda_fail(regmem_t* h, cudaError_t e, const char* what) {
  return fail(h, REGMEM_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define RM_CUDA(h, call)                                  \
  do {                                                    \
    cudaError_t e_ = (call);                              \
    if (e_ != cudaSuccess) return cuda_fail((h), e_, #call); \
  } while (0)

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
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

// Frame tensor [N][H][64] bf16 viewed as 3-D (channel, head, token); one box is
// one head's 128 consecutive tokens, 128-byte swizzled.
bool encode_frame_map(CUtensorMap* m, const void* ptr, int N, int H) {
  auto enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)H, (cuuint64_t)N};
  cuuint64_t strides[2] = {(cuuint64_t)kHeadDim * 2, (cuuint64_t)H * kHeadDim * 2};
  cuuint32_t box[3] = {(cuuint32_t)kHeadDim, 1, (cuuint32_t)kTile};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

// Bank [H][cap][64] bf16 viewed as 3-D (channel, row, head); one box is 128
// rows of one head.
bool encode_bank_map(CUtensorMap* m, const void* ptr, long long cap, int H) {
  auto enc = encode_fn();
  if (!enc) return false;
  cuuint64_t dims[3] = {(cuuint64_t)kHeadDim, (cuuint64_t)cap, (cuuint64_t)H};
  cuuint64_t strides[2] = {(cuuint64_t)kHeadDim * 2, (cuuint64_t)cap * kHeadDim * 2};
  cuuint32_t box[3] = {(cuuint32_t)kHeadDim, (cuuint32_t)kTile, 1};
  cuuint32_t es[3] = {1, 1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(ptr), dims, strides, box, es,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

regmem_status check_device_status(regmem_t* h) {
  if (h->status_host && *reinterpret_cast<volatile int*>(h->status_host) != 0) {
    const int s = *reinterpret_cast<volatile int*>(h->status_host);
    if (s & kStatusRange)
      return fail(h, REGMEM_ERR_DEVICE_CHECK,
                  "a kernel reported device status 0x%x (a range guard of the checked build "
                  "failed); destroy the handle", s);
    return fail(h, REGMEM_ERR_TIMEOUT,
                "a kernel reported device status 0x%x (%s); destroy the handle", s,
                (s & kStatusTimeout) ? "bounded wait expired" : "shared-memory alignment");
  }
  return REGMEM_OK;
}

regmem_status ready(regmem_t* h, int layer, bool need_layer) {
  if (!h) return REGMEM_ERR_ARG;
  if (!h->frame_set) return fail(h, REGMEM_ERR_STATE, "regmem_set_frame has not been called");
  if (need_layer && (layer < 0 || layer >= h->layers))
    return fail(h, REGMEM_ERR_ARG, "layer %d out of range [0, %d)", layer, h->layers);
  regmem_status s = check_device_status(h);
  if (s != REGMEM_OK) return s;
  if (cudaSetDevice(h->device) != cudaSuccess)
    return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
  return REGMEM_OK;
}

constexpr size_t kEventPairs = 256;
constexpr long long kClockSlots = 1 << 20;  // launches one profiling window can clock (16 MB)

// Adds the elapsed times of event triple i to the profile and frees the slot.
cudaError_t harvest_pair(regmem_t* h, size_t i) {
  cudaError_t e = cudaEventSynchronize(h->ev_ring[3 * i + 2]);
  if (e != cudaSuccess) return e;
  float ms = 0.f, ms2 = 0.f;
  e = cudaEventElapsedTime(&ms, h->ev_ring[3 * i], h->ev_ring[3 * i + 1]);
  if (e != cudaSuccess) return e;
  e = cudaEventElapsedTime(&ms2, h->ev_ring[3 * i + 1], h->ev_ring[3 * i + 2]);
  if (e != cudaSuccess) return e;
  h->prof.attention_ms += ms;
  h->prof.merge_ms += ms2;
  h->ev_busy[i] = 0;
  return cudaSuccess;
}

float* lse_of(regmem_t* h, int layer) { return h->lse + (size_t)layer * h->heads * h->N; }

// Orders the handle's stream after every side submission so far.
regmem_status join_side(regmem_t* h) {
  if (h->side_seq > h->covered_seq) {
    RM_CUDA(h, cudaStreamWaitEvent(h->stream, h->side_ev, 0));
    h->covered_seq = h->side_seq;
  }
  return REGMEM_OK;
}

regmem_status run_attention(regmem_t* h, int layer, const void* Q, const void* K, const void* V,
                            void* out, int M, bool frame_attention = false) {
  // the layer's previous saliency and admission (side stream) read its LSE
  // rows and append to its bank: they finish before this attention starts.
  // One wait covers all side work so far, so in a stream of frames only the
  // first layer of each frame waits.
  if (h->side_seq_of[layer] > h->covered_seq) {
    regmem_status s = join_side(h);
    if (s != REGMEM_OK) return s;
  }
  CUtensorMap tq, tk, tv;
  if (!encode_frame_map(&tq, Q, h->N, h->heads) || !encode_frame_map(&tk, K, h->N, h->heads) ||
      !encode_frame_map(&tv, V, h->N, h->heads))
    return fail(h, REGMEM_ERR_CUDA, "cuTensorMapEncodeTiled failed for the frame tensors");
  AttnArgs a = {};
  a.tmQ = &tq;
  a.tmK = &tk;
  a.tmV = &tv;
  a.tmBK = &h->tmBK[layer];
  a.tmBV = &h->tmBV[layer];
  a.N = h->N;
  a.H = h->heads;
  a.M = M;
  a.scale = h->scale;
  a.out = static_cast<__nv_bfloat16*>(out);
  a.lse = lse_of(h, layer);
  h->lse_layer = layer;
  a.part_o = h->part_o;
  a.part_lse = h->part_lse;
  a.max_phases = kAttnMaxPhases;
  a.status = h->status_dev;
  a.wait_ns = h->wait_ns;
  a.fault_skip_kv = h->fault_skip_kv;
  h->fault_skip_kv = -1;  // one launch only
  if (h->kclock && h->time_every > 0 && h->clk_next < kClockSlots) {
    a.clk_start = h->kclock + h->clk_next;
    a.clk_end = h->kclock + kClockSlots + h->clk_next;
    h->clk_frame[h->clk_next] = frame_attention ? 1 : 0;
    ++h->clk_next;
  }
  const AttnPlan pl = attn_plan(h->N, h->heads, M);
  const long long G = pl.total < h->attn_grid ? pl.total : h->attn_grid;
  a.grid = (int)G;
  cudaEvent_t eb = nullptr, ea = nullptr, em = nullptr;
  const bool timed = h->time_every > 0 && h->attn_launch_no % h->time_every == 0;
  ++h->attn_launch_no;
  if (timed) {
    if (h->ev_ring.empty()) {
      h->ev_ring.resize(3 * kEventPairs);
      h->ev_busy.assign(kEventPairs, 0);
      for (auto& e : h->ev_ring) RM_CUDA(h, cudaEventCreate(&e));
    }
    const size_t i = h->ev_next;
    if (h->ev_busy[i]) RM_CUDA(h, harvest_pair(h, i));
    eb = h->ev_ring[3 * i];
    ea = h->ev_ring[3 * i + 1];
    em = h->ev_ring[3 * i + 2];
    h->ev_busy[i] = 1;
    h->ev_next = (i + 1) % kEventPairs;
  }
  RM_CUDA(h, launch_attention(a, h->stream, eb, ea, em));
  h->prof.attention_ctas = a.grid;
  h->prof.attention_ctas_per_sm = h->attn_ctas_per_sm;
  const double L = (double)M + h->N;
  h->prof.launches_attention += 1;
  if (a.grid > 1) h->prof.launches_combine += 1;
  if (frame_attention) h->prof.launches_frame_attention += 1;
  if (a.clk_start) {
    const double flops = 4.0 * h->N * L * kHeadDim * h->heads;
    if (frame_attention) h->prof.frame_attention_clock_flops += flops;
    else h->prof.attention_clock_flops += flops;
  }
  if (timed) {
    h->prof.attention_timed += 1;
    h->prof.attention_flops += 4.0 * h->N * L * kHeadDim * h->heads;
    h->prof.attention_bytes += (2.0 * h->N * h->heads * kHeadDim * 2)   // Q in, O out
                               + (2.0 * L * h->heads * kHeadDim * 2)    // K and V rows
                               + (4.0 * h->heads * h->N);               // LSE
  }
  return REGMEM_OK;
}

}  // namespace

extern "C" {

const char* regmem_status_string(regmem_status s) {
  switch (s) {
    case REGMEM_OK: return "REGMEM_OK";
    case REGMEM_ERR_ARG: return "REGMEM_ERR_ARG";
    case REGMEM_ERR_STATE: return "REGMEM_ERR_STATE";
    case REGMEM_ERR_CAPACITY: return "REGMEM_ERR_CAPACITY";
    case REGMEM_ERR_CUDA: return "REGMEM_ERR_CUDA";
    case REGMEM_ERR_UNSUPPORTED: return "REGMEM_ERR_UNSUPPORTED";
    case REGMEM_ERR_TIMEOUT: return "REGMEM_ERR_TIMEOUT";
    case REGMEM_ERR_DEVICE_CHECK: return "REGMEM_ERR_DEVICE_CHECK";
  }
  return "REGMEM_UNKNOWN";
}

const char* regmem_last_error(const regmem_t* h) { return h ? h->err.c_str() : "null handle"; }

regmem_status regmem_create(regmem_t** out, int32_t layers, int32_t heads, int32_t head_dim,
                            int32_t budget) {
  if (!out) return REGMEM_ERR_ARG;
  *out = nullptr;
  if (layers < 1 || heads < 1 || budget < 0) return REGMEM_ERR_ARG;
  if (head_dim != kHeadDim) return REGMEM_ERR_UNSUPPORTED;
  regmem_t* h = new (std::nothrow) regmem_t();
  if (!h) return REGMEM_ERR_ARG;
  h->layers = layers;
  h->heads = heads;
  h->head_dim = head_dim;
  h->budget = budget;
  h->len.assign(layers, 0);
  h->pending.assign(layers, 0);
  h->pK.assign(layers, nullptr);
  h->pV.assign(layers, nullptr);
  h->pS.assign(layers, nullptr);
  h->stK.assign(layers, nullptr);
  h->stV.assign(layers, nullptr);
  h->side_seq_of.assign(layers, 0);
  *out = h;
  return REGMEM_OK;
}

namespace {

// Staging buffers, copy streams and events of the host-buffer entry points:
// the six sets of regmem_attend_admit_host, and Q / out / saliency plus
// per-layer K and V (kept until the layer's admit) of
// regmem_attend_frame_host.  Made once, by regmem_set_frame, so that no
// host-buffer call allocates (a cudaMalloc inside a stream of calls would
// synchronise the device and stall the copies' overlap).
regmem_status alloc_staging(regmem_t* h) {
  const size_t tbytes = (size_t)h->N * h->heads * kHeadDim * 2;
  const size_t sbytes = (size_t)h->heads * h->N * sizeof(float);
  RM_CUDA(h, cudaStreamCreateWithFlags(&h->cstream, cudaStreamNonBlocking));
  RM_CUDA(h, cudaStreamCreateWithFlags(&h->dstream, cudaStreamNonBlocking));
  for (auto& hs : h->hs) {
    RM_CUDA(h, cudaMalloc(&hs.q, tbytes));
    RM_CUDA(h, cudaMalloc(&hs.k, tbytes));
    RM_CUDA(h, cudaMalloc(&hs.v, tbytes));
    RM_CUDA(h, cudaMalloc(&hs.out, tbytes));
    RM_CUDA(h, cudaMalloc(&hs.sal, sbytes));
    RM_CUDA(h, cudaEventCreateWithFlags(&hs.h2d, cudaEventDisableTiming));
    RM_CUDA(h, cudaEventCreateWithFlags(&hs.done, cudaEventDisableTiming));
    RM_CUDA(h, cudaEventCreateWithFlags(&hs.d2h, cudaEventDisableTiming));
  }
  RM_CUDA(h, cudaMalloc(&h->stQ, tbytes));
  RM_CUDA(h, cudaMalloc(&h->stOut, tbytes));
  RM_CUDA(h, cudaMalloc(&h->stSal, sbytes));
  for (int l = 0; l < h->layers; ++l) {
    RM_CUDA(h, cudaMalloc(&h->stK[l], tbytes));
    RM_CUDA(h, cudaMalloc(&h->stV[l], tbytes));
  }
  return REGMEM_OK;
}

}  // namespace

regmem_status regmem_set_frame(regmem_t* h, const regmem_frame_desc* fd) {
  REGMEM_RANGE;
  if (!h || !fd) return REGMEM_ERR_ARG;
  if (h->frame_set) return fail(h, REGMEM_ERR_STATE, "frame geometry already set");
  const int ds = fd->ds == 0 ? 2 : fd->ds;
  if (fd->n_special < 0 || fd->grid_h < 1 || fd->grid_w < 1 || ds < 1 || fd->max_frames < 1 ||
      fd->n_tokens != fd->n_special + fd->grid_h * fd->grid_w || fd->scale < 0.f ||
      !std::isfinite(fd->scale) || (fd->candidates != 0 && fd->candidates != 1))
    return fail(h, REGMEM_ERR_ARG, "inconsistent frame descriptor");
  const int N = fd->n_tokens;
  if (N > 65536) return fail(h, REGMEM_ERR_UNSUPPORTED, "n_tokens %d > 65536", N);
  const int cand_lo = fd->candidates == 0 ? fd->n_special : 0;
  if (N - cand_lo > kMaxCandidates)
    return fail(h, REGMEM_ERR_UNSUPPORTED, "%d admission candidates > %d", N - cand_lo,
                kMaxCandidates);
  // sampled queries: top-left of each ds x ds window of the patch grid
  std::vector<int> q;
  for (int r = 0; r < fd->grid_h; r += ds)
    for (int c = 0; c < fd->grid_w; c += ds) q.push_back(fd->n_special + r * fd->grid_w + c);
  if ((int)q.size() > 8192) return fail(h, REGMEM_ERR_UNSUPPORTED, "too many sampled queries");
  const long long cap = (long long)N + (long long)(fd->max_frames - 1) * h->budget;
  if (cap > (1LL << 31) - 1) return fail(h, REGMEM_ERR_UNSUPPORTED, "bank capacity too large");

  RM_CUDA(h, cudaGetDevice(&h->device));
  int sms = 0;
  RM_CUDA(h, cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, h->device));
  RM_CUDA(h, attn_setup());
  RM_CUDA(h, saliency_setup());
  RM_CUDA(h, admit_setup());
  if (!encode_fn()) return fail(h, REGMEM_ERR_CUDA, "cuTensorMapEncodeTiled entry point missing");

  const size_t bank_elems = (size_t)h->layers * h->heads * cap * kHeadDim;
  h->attn_ctas_per_sm = attn_ctas_per_sm();
  h->attn_grid = std::min(sms * h->attn_ctas_per_sm, kAttnMaxGrid);
  RM_CUDA(h, cudaMalloc(&h->bankK, bank_elems * 2));
  RM_CUDA(h, cudaMalloc(&h->bankV, bank_elems * 2));
  RM_CUDA(h, cudaMemset(h->bankK, 0, bank_elems * 2));
  RM_CUDA(h, cudaMemset(h->bankV, 0, bank_elems * 2));
  RM_CUDA(h, cudaMalloc(&h->lse, (size_t)h->layers * h->heads * N * sizeof(float)));
  RM_CUDA(h, cudaMalloc(&h->qidx, q.size() * sizeof(int) + 4));
  RM_CUDA(h, cudaMemcpy(h->qidx, q.data(), q.size() * sizeof(int), cudaMemcpyHostToDevice));
  RM_CUDA(h, cudaMalloc(&h->part_o, attn_part_o_elems(h->attn_grid, kAttnMaxPhases) * sizeof(__nv_bfloat16)));
  RM_CUDA(h, cudaMalloc(&h->part_lse, attn_part_lse_floats(h->attn_grid, kAttnMaxPhases) * sizeof(float)));
  {  // per-head counters, or per key tile plus one (the shared selection)
    const size_t nd = std::max(h->heads, (N + kTile - 1) / kTile + 1);
    RM_CUDA(h, cudaMalloc(&h->head_done, nd * sizeof(int)));
    RM_CUDA(h, cudaMemset(h->head_done, 0, nd * sizeof(int)));
  }
  RM_CUDA(h, cudaMalloc(&h->adm_lists, (size_t)h->heads * ((N + kTile - 1) / kTile) * 32 * sizeof(uint64_t)));
  RM_CUDA(h, cudaHostAlloc(&h->status_host, sizeof(int), cudaHostAllocMapped));
  *h->status_host = 0;
  RM_CUDA(h, cudaHostGetDevicePointer(&h->status_dev, h->status_host, 0));

  h->tmBK.resize(h->layers);
  h->tmBV.resize(h->layers);
  for (int l = 0; l < h->layers; ++l) {
    const size_t off = (size_t)l * h->heads * cap * kHeadDim;
    if (!encode_bank_map(&h->tmBK[l], h->bankK + off, cap, h->heads) ||
        !encode_bank_map(&h->tmBV[l], h->bankV + off, cap, h->heads))
      return fail(h, REGMEM_ERR_CUDA, "cuTensorMapEncodeTiled failed for the bank");
  }
  h->N = N;
  h->n_special = fd->n_special;
  h->grid_h = fd->grid_h;
  h->grid_w = fd->grid_w;
  h->ds = ds;
  h->cand_lo = cand_lo;
  h->nq = (int)q.size();
  h->max_frames = fd->max_frames;
  h->scale = fd->scale == 0.f ? 1.f / std::sqrt((float)h->head_dim) : fd->scale;
  h->cap = cap;
  regmem_status s = alloc_staging(h);
  if (s != REGMEM_OK) return s;
  h->frame_set = true;
  return REGMEM_OK;
}

regmem_status regmem_set_overlap(regmem_t* h, int32_t on) {
  REGMEM_RANGE;
  if (!h || (on != 0 && on != 1)) return REGMEM_ERR_ARG;
  if (!on && h->frame_set && h->side_seq > h->covered_seq) {
    if (cudaSetDevice(h->device) != cudaSuccess)
      return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
    regmem_status s = join_side(h);
    if (s != REGMEM_OK) return s;
  }
  h->overlap = on != 0;
  return REGMEM_OK;
}

regmem_status regmem_join(regmem_t* h) {
  REGMEM_RANGE;
  if (!h) return REGMEM_ERR_ARG;
  if (!h->frame_set || h->side_seq <= h->covered_seq) return REGMEM_OK;
  if (cudaSetDevice(h->device) != cudaSuccess)
    return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
  return join_side(h);
}

regmem_status regmem_set_stream(regmem_t* h, void* stream) {
  if (!h) return REGMEM_ERR_ARG;
  h->stream = static_cast<cudaStream_t>(stream);
  h->covered_seq = 0;  // the new stream has waited for no side work yet
  return REGMEM_OK;
}

namespace {

// Attention and saliency of one frame on one layer; with `adm` the saliency
// kernel also runs the admission of adm->k rows per head (fused path).
regmem_status attend_impl(regmem_t* h, int32_t layer, const void* Q, const void* K, const void* V,
                          void* out, float* saliency, const AdmitArgs* adm, cudaStream_t sst) {
  const long long M = h->len[layer];
  regmem_status s = run_attention(h, layer, Q, K, V, out, (int)M);
  if (s != REGMEM_OK) return s;
  if (sst != h->stream) {  // the side work starts once the attention (and its merge) is done
    RM_CUDA(h, cudaEventRecord(h->main_ev, h->stream));
    RM_CUDA(h, cudaStreamWaitEvent(sst, h->main_ev, 0));
  }
  CUtensorMap tk;
  if (!encode_frame_map(&tk, K, h->N, h->heads))
    return fail(h, REGMEM_ERR_CUDA, "cuTensorMapEncodeTiled failed for K");
  SalArgs sa = {};
  sa.tmK = &tk;
  sa.Q = static_cast<const __nv_bfloat16*>(Q);
  sa.qidx = h->qidx;
  sa.nq = h->nq;
  sa.lse = lse_of(h, layer);
  sa.N = h->N;
  sa.H = h->heads;
  sa.scale = h->scale;
  sa.sal = saliency;
  sa.status = h->status_dev;
  sa.adm = adm;
  RM_CUDA(h, launch_saliency(sa, sst));
  h->prof.launches_saliency += 1;
  return REGMEM_OK;
}

regmem_status check_tensors(regmem_t* h, const void* Q, const void* K, const void* V,
                            const void* out, const float* saliency) {
  if (!Q || !K || !V || !out || !saliency)
    return fail(h, REGMEM_ERR_ARG, "null tensor pointer");
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(out) || !aligned16(saliency))
    return fail(h, REGMEM_ERR_ARG, "tensor pointers must be 16-byte aligned");
  return REGMEM_OK;
}

// k range and capacity of an admission on a non-empty layer.
regmem_status check_admit(regmem_t* h, int32_t layer, int32_t k) {
  const int nc = h->N - h->cand_lo;
  const int kmax = h->budget < nc ? h->budget : nc;
  if (k < 0 || k > kmax)
    return fail(h, REGMEM_ERR_ARG, "k = %d outside [0, %d] (budget %d, candidates %d)", k, kmax,
                h->budget, nc);
  if (h->len[layer] + k > h->cap)
    return fail(h, REGMEM_ERR_CAPACITY, "layer %d: %lld + %d rows exceed capacity %lld", layer,
                h->len[layer], k, h->cap);
  return REGMEM_OK;
}

AdmitArgs admit_args(regmem_t* h, int32_t layer, const void* K, const void* V, float* saliency,
                     int32_t k, int32_t* idx_out) {
  AdmitArgs a = {};
  a.sal = saliency;
  a.K = static_cast<const __nv_bfloat16*>(K);
  a.V = static_cast<const __nv_bfloat16*>(V);
  a.bankK = h->bankK + (size_t)layer * h->heads * h->cap * kHeadDim;
  a.bankV = h->bankV + (size_t)layer * h->heads * h->cap * kHeadDim;
  a.cap = h->cap;
  a.M = h->len[layer];
  a.N = h->N;
  a.H = h->heads;
  a.cand_lo = h->cand_lo;
  a.k = k;
  a.idx_out = idx_out;
  a.lists = h->adm_lists;
  a.done = h->head_done;
  a.status = h->status_dev;
  return a;
}

// Creates the side stream (lowest priority, so that the attention's CTAs are
// dispatched ahead of its blocks when both wait for SMs) and its events.
regmem_status side_stream(regmem_t* h) {
  if (h->sstream) return REGMEM_OK;
  int least = 0, greatest = 0;
  RM_CUDA(h, cudaDeviceGetStreamPriorityRange(&least, &greatest));
  RM_CUDA(h, cudaStreamCreateWithPriority(&h->sstream, cudaStreamNonBlocking, least));
  RM_CUDA(h, cudaEventCreateWithFlags(&h->main_ev, cudaEventDisableTiming));
  RM_CUDA(h, cudaEventCreateWithFlags(&h->side_ev, cudaEventDisableTiming));
  return REGMEM_OK;
}

// Marks the end of a layer's side submission on stream sst.
regmem_status finish_side(regmem_t* h, int layer, cudaStream_t sst) {
  if (sst == h->stream) return REGMEM_OK;
  RM_CUDA(h, cudaEventRecord(h->side_ev, sst));
  h->side_seq_of[layer] = ++h->side_seq;
  return REGMEM_OK;
}

}  // namespace

regmem_status regmem_attend_frame(regmem_t* h, int32_t layer, const void* Q, const void* K,
                                  const void* V, void* out, float* saliency) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if ((s = check_tensors(h, Q, K, V, out, saliency)) != REGMEM_OK) return s;
  if (h->pending[layer])
    return fail(h, REGMEM_ERR_STATE, "layer %d already has an attend pending; call regmem_admit",
                layer);
  // the two-call path runs on the handle's stream and shares the selection
  // scratch with side-stream admissions
  if ((s = join_side(h)) != REGMEM_OK) return s;
  if ((s = attend_impl(h, layer, Q, K, V, out, saliency, nullptr, h->stream)) != REGMEM_OK) return s;
  h->pending[layer] = 1;
  h->pK[layer] = static_cast<const __nv_bfloat16*>(K);
  h->pV[layer] = static_cast<const __nv_bfloat16*>(V);
  h->pS[layer] = saliency;
  return REGMEM_OK;
}

namespace {

// regmem_attend_admit and regmem_attend_admit_shared: the attention on the
// handle's stream, then the saliency and the selection (per head, fused into
// the saliency kernel for k <= 32, or head-averaged) and the append on the
// side stream when overlap is on.
regmem_status attend_admit_impl(regmem_t* h, int32_t layer, const void* Q, const void* K,
                                const void* V, void* out, float* saliency, int32_t k,
                                int32_t* idx_out, bool shared) {
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if ((s = check_tensors(h, Q, K, V, out, saliency)) != REGMEM_OK) return s;
  if (h->pending[layer])
    return fail(h, REGMEM_ERR_STATE, "layer %d already has an attend pending; call regmem_admit",
                layer);
  if (idx_out && ((reinterpret_cast<uintptr_t>(idx_out) & 3u) != 0))
    return fail(h, REGMEM_ERR_ARG, "idx_out must be 4-byte aligned");
  cudaStream_t sst = h->stream;  // stream of the saliency and admission
  if (h->overlap) {
    if ((s = side_stream(h)) != REGMEM_OK) return s;
    sst = h->sstream;
  }
  if (h->len[layer] == 0) {  // Eq. 4: the first frame is kept whole
    if ((s = attend_impl(h, layer, Q, K, V, out, saliency, nullptr, sst)) != REGMEM_OK) return s;
    auto* bk = h->bankK + (size_t)layer * h->heads * h->cap * kHeadDim;
    auto* bv = h->bankV + (size_t)layer * h->heads * h->cap * kHeadDim;
    RM_CUDA(h, launch_anchor(static_cast<const __nv_bfloat16*>(K), static_cast<const __nv_bfloat16*>(V),
                             bk, bv, h->cap, h->N, h->heads, h->status_dev, sst));
    h->prof.launches_anchor += 1;
    h->len[layer] = h->N;
    return finish_side(h, layer, sst);
  }
  if ((s = check_admit(h, layer, k)) != REGMEM_OK) return s;
  AdmitArgs a = admit_args(h, layer, K, V, saliency, k, idx_out);
  a.shared = shared ? 1 : 0;
  // k <= 32: the admission (per head, or head-averaged) runs inside the
  // saliency kernel; larger k takes a selection kernel of its own
  const bool fused = k > 0 && k <= kFusedMaxK;
  if ((s = attend_impl(h, layer, Q, K, V, out, saliency, fused ? &a : nullptr, sst)) != REGMEM_OK)
    return s;
  if (k > 0 && !fused) {
    RM_CUDA(h, shared ? launch_admit_shared(a, sst) : launch_admit(a, sst));
    h->prof.launches_admit += 1;
  }
  h->len[layer] += k;
  return finish_side(h, layer, sst);
}

}  // namespace

regmem_status regmem_attend_admit(regmem_t* h, int32_t layer, const void* Q, const void* K,
                                  const void* V, void* out, float* saliency, int32_t k,
                                  int32_t* idx_out) {
  REGMEM_RANGE;
  return attend_admit_impl(h, layer, Q, K, V, out, saliency, k, idx_out, false);
}

regmem_status regmem_attend_admit_shared(regmem_t* h, int32_t layer, const void* Q, const void* K,
                                         const void* V, void* out, float* saliency, int32_t k,
                                         int32_t* idx_out) {
  REGMEM_RANGE;
  return attend_admit_impl(h, layer, Q, K, V, out, saliency, k, idx_out, true);
}

namespace {

// Copies a frame's Q, K, V from host memory into the handle's staging buffers
// (K and V per layer: they must stay valid until the layer's admission).
regmem_status stage_inputs(regmem_t* h, int32_t layer, const void* hostQ, const void* hostK,
                           const void* hostV) {
  const size_t tbytes = (size_t)h->N * h->heads * kHeadDim * 2;
  RM_CUDA(h, cudaMemcpyAsync(h->stQ, hostQ, tbytes, cudaMemcpyHostToDevice, h->stream));
  RM_CUDA(h, cudaMemcpyAsync(h->stK[layer], hostK, tbytes, cudaMemcpyHostToDevice, h->stream));
  RM_CUDA(h, cudaMemcpyAsync(h->stV[layer], hostV, tbytes, cudaMemcpyHostToDevice, h->stream));
  return REGMEM_OK;
}

regmem_status unstage_outputs(regmem_t* h, void* hostOut, float* hostSaliency) {
  const size_t tbytes = (size_t)h->N * h->heads * kHeadDim * 2;
  const size_t sbytes = (size_t)h->heads * h->N * sizeof(float);
  RM_CUDA(h, cudaMemcpyAsync(hostOut, h->stOut, tbytes, cudaMemcpyDeviceToHost, h->stream));
  RM_CUDA(h, cudaMemcpyAsync(hostSaliency, h->stSal, sbytes, cudaMemcpyDeviceToHost, h->stream));
  return REGMEM_OK;
}

}  // namespace

regmem_status regmem_attend_frame_host(regmem_t* h, int32_t layer, const void* hostQ,
                                       const void* hostK, const void* hostV, void* hostOut,
                                       float* hostSaliency) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if (!hostQ || !hostK || !hostV || !hostOut || !hostSaliency)
    return fail(h, REGMEM_ERR_ARG, "null host pointer");
  if (h->pending[layer])
    return fail(h, REGMEM_ERR_STATE, "layer %d already has an attend pending; call regmem_admit",
                layer);
  if ((s = stage_inputs(h, layer, hostQ, hostK, hostV)) != REGMEM_OK) return s;
  s = regmem_attend_frame(h, layer, h->stQ, h->stK[layer], h->stV[layer], h->stOut, h->stSal);
  if (s != REGMEM_OK) return s;
  return unstage_outputs(h, hostOut, hostSaliency);
}

regmem_status regmem_attend_admit_host(regmem_t* h, int32_t layer, const void* hostQ,
                                       const void* hostK, const void* hostV, void* hostOut,
                                       float* hostSaliency, int32_t k) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if (!hostQ || !hostK || !hostV || !hostOut || !hostSaliency)
    return fail(h, REGMEM_ERR_ARG, "null host pointer");
  if (h->pending[layer])
    return fail(h, REGMEM_ERR_STATE, "layer %d already has an attend pending; call regmem_admit",
                layer);
  if (h->len[layer] > 0 && (s = check_admit(h, layer, k)) != REGMEM_OK) return s;
  // Staging set b (in turn): its inputs are copied in on the input copy
  // stream once the kernels of its previous use are done, the kernels run on
  // the handle's stream once the inputs are in and the previous outputs out,
  // and the outputs are copied back on the output copy stream.  The two copy
  // streams are separate so that the next call's inputs need not wait for
  // this call's outputs: its copies overlap this call's kernels.
  regmem_t::HostSet& hs = h->hs[h->hs_next % regmem_t::kHostSets];
  ++h->hs_next;
  const size_t tbytes = (size_t)h->N * h->heads * kHeadDim * 2;
  const size_t sbytes = (size_t)h->heads * h->N * sizeof(float);
  // The input copy stream also waits for the set's previous output copies,
  // so that the handle's stream needs one event wait per call (each wait
  // between two kernels costs the launch overlap of the second).
  if (hs.used) {
    RM_CUDA(h, cudaStreamWaitEvent(h->cstream, hs.done, 0));
    RM_CUDA(h, cudaStreamWaitEvent(h->cstream, hs.d2h, 0));
  }
  RM_CUDA(h, cudaMemcpyAsync(hs.q, hostQ, tbytes, cudaMemcpyHostToDevice, h->cstream));
  RM_CUDA(h, cudaMemcpyAsync(hs.k, hostK, tbytes, cudaMemcpyHostToDevice, h->cstream));
  RM_CUDA(h, cudaMemcpyAsync(hs.v, hostV, tbytes, cudaMemcpyHostToDevice, h->cstream));
  RM_CUDA(h, cudaEventRecord(hs.h2d, h->cstream));
  RM_CUDA(h, cudaStreamWaitEvent(h->stream, hs.h2d, 0));
  s = regmem_attend_admit(h, layer, hs.q, hs.k, hs.v, hs.out, hs.sal, k, nullptr);
  if (s != REGMEM_OK) return s;
  // with overlap the call ends on the side stream (its saliency and
  // admission follow the attention there)
  RM_CUDA(h, cudaEventRecord(hs.done, h->overlap ? h->sstream : h->stream));
  RM_CUDA(h, cudaStreamWaitEvent(h->dstream, hs.done, 0));
  RM_CUDA(h, cudaMemcpyAsync(hostOut, hs.out, tbytes, cudaMemcpyDeviceToHost, h->dstream));
  RM_CUDA(h, cudaMemcpyAsync(hostSaliency, hs.sal, sbytes, cudaMemcpyDeviceToHost, h->dstream));
  RM_CUDA(h, cudaEventRecord(hs.d2h, h->dstream));
  hs.used = true;
  return REGMEM_OK;
}

regmem_status regmem_admit(regmem_t* h, int32_t layer, int32_t k, int32_t* idx_out) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if (!h->pending[layer])
    return fail(h, REGMEM_ERR_STATE, "layer %d has no attend pending", layer);
  if (idx_out && ((reinterpret_cast<uintptr_t>(idx_out) & 3u) != 0))
    return fail(h, REGMEM_ERR_ARG, "idx_out must be 4-byte aligned");
  if (h->len[layer] == 0) {  // Eq. 4: the first frame is kept whole
    auto* bk = h->bankK + (size_t)layer * h->heads * h->cap * kHeadDim;
    auto* bv = h->bankV + (size_t)layer * h->heads * h->cap * kHeadDim;
    RM_CUDA(h, launch_anchor(h->pK[layer], h->pV[layer], bk, bv, h->cap, h->N, h->heads, h->status_dev,
                             h->stream));
    h->prof.launches_anchor += 1;
    h->len[layer] = h->N;
    h->pending[layer] = 0;
    return REGMEM_OK;
  }
  if ((s = check_admit(h, layer, k)) != REGMEM_OK) return s;
  if (k > 0) {
    const AdmitArgs a = admit_args(h, layer, h->pK[layer], h->pV[layer], h->pS[layer], k, idx_out);
    RM_CUDA(h, launch_admit(a, h->stream));
    h->prof.launches_admit += 1;
  }
  h->len[layer] += k;
  h->pending[layer] = 0;
  return REGMEM_OK;
}

regmem_status regmem_admit_shared(regmem_t* h, int32_t layer, int32_t k, int32_t* idx_out) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if (!h->pending[layer])
    return fail(h, REGMEM_ERR_STATE, "layer %d has no attend pending", layer);
  if (idx_out && ((reinterpret_cast<uintptr_t>(idx_out) & 3u) != 0))
    return fail(h, REGMEM_ERR_ARG, "idx_out must be 4-byte aligned");
  if (h->len[layer] == 0) return regmem_admit(h, layer, k, nullptr);  // Eq. 4 anchor
  if ((s = check_admit(h, layer, k)) != REGMEM_OK) return s;
  if (k > 0) {
    const AdmitArgs a = admit_args(h, layer, h->pK[layer], h->pV[layer], h->pS[layer], k, idx_out);
    RM_CUDA(h, launch_admit_shared(a, h->stream));
    h->prof.launches_admit += 1;
  }
  h->len[layer] += k;
  h->pending[layer] = 0;
  return REGMEM_OK;
}

regmem_status regmem_frame_attention(regmem_t* h, const void* Q, const void* K, const void* V,
                                     void* out) {
  REGMEM_RANGE;
  regmem_status s = ready(h, 0, false);
  if (s != REGMEM_OK) return s;
  if (!Q || !K || !V || !out) return fail(h, REGMEM_ERR_ARG, "null tensor pointer");
  if (!aligned16(Q) || !aligned16(K) || !aligned16(V) || !aligned16(out))
    return fail(h, REGMEM_ERR_ARG, "tensor pointers must be 16-byte aligned");
  return run_attention(h, 0, Q, K, V, out, 0, true);
}

regmem_status regmem_reset(regmem_t* h) {
  REGMEM_RANGE;
  if (!h) return REGMEM_ERR_ARG;
  if (h->frame_set && h->side_seq > h->covered_seq) {  // the new stream's writes follow the old side work
    if (cudaSetDevice(h->device) != cudaSuccess)
      return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
    regmem_status s = join_side(h);
    if (s != REGMEM_OK) return s;
  }
  for (int l = 0; l < h->layers; ++l) {
    h->len[l] = 0;
    h->pending[l] = 0;
  }
  return REGMEM_OK;
}

regmem_status regmem_memory_len(const regmem_t* h, int32_t layer, int64_t* len) {
  if (!h || !len || layer < 0 || layer >= h->layers) return REGMEM_ERR_ARG;
  *len = h->len[layer];
  return REGMEM_OK;
}

regmem_status regmem_capacity(const regmem_t* h, int64_t* rows) {
  if (!h || !rows) return REGMEM_ERR_ARG;
  if (!h->frame_set) return REGMEM_ERR_STATE;
  *rows = h->cap;
  return REGMEM_OK;
}

regmem_status regmem_export_bank(regmem_t* h, int32_t layer, void* hostK, void* hostV) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if (!hostK || !hostV) return fail(h, REGMEM_ERR_ARG, "null host pointer");
  const long long n = h->len[layer];
  if (n == 0) return REGMEM_OK;
  const size_t row = kHeadDim * 2;
  const size_t off = (size_t)layer * h->heads * h->cap * kHeadDim;
  if ((s = join_side(h)) != REGMEM_OK) return s;  // admissions still appending on the side stream
  RM_CUDA(h, cudaMemcpy2DAsync(hostK, n * row, h->bankK + off, h->cap * row, n * row, h->heads,
                               cudaMemcpyDeviceToHost, h->stream));
  RM_CUDA(h, cudaMemcpy2DAsync(hostV, n * row, h->bankV + off, h->cap * row, n * row, h->heads,
                               cudaMemcpyDeviceToHost, h->stream));
  RM_CUDA(h, cudaStreamSynchronize(h->stream));
  return check_device_status(h);
}

regmem_status regmem_import_bank(regmem_t* h, int32_t layer, const void* hostK, const void* hostV,
                                 int64_t len) {
  REGMEM_RANGE;
  regmem_status s = ready(h, layer, true);
  if (s != REGMEM_OK) return s;
  if (len < 0 || len > h->cap)
    return fail(h, REGMEM_ERR_CAPACITY, "len %lld outside [0, %lld]", (long long)len, h->cap);
  if (len > 0 && (!hostK || !hostV)) return fail(h, REGMEM_ERR_ARG, "null host pointer");
  const size_t row = kHeadDim * 2;
  const size_t off = (size_t)layer * h->heads * h->cap * kHeadDim;
  if ((s = join_side(h)) != REGMEM_OK) return s;
  if (len > 0) {
    RM_CUDA(h, cudaMemcpy2DAsync(h->bankK + off, h->cap * row, hostK, len * row, len * row,
                                 h->heads, cudaMemcpyHostToDevice, h->stream));
    RM_CUDA(h, cudaMemcpy2DAsync(h->bankV + off, h->cap * row, hostV, len * row, len * row,
                                 h->heads, cudaMemcpyHostToDevice, h->stream));
  }
  RM_CUDA(h, cudaStreamSynchronize(h->stream));
  h->len[layer] = len;
  h->pending[layer] = 0;
  return REGMEM_OK;
}

regmem_status regmem_copy_lse(regmem_t* h, float* dst) {
  REGMEM_RANGE;
  regmem_status s = ready(h, 0, false);
  if (s != REGMEM_OK) return s;
  if (!dst) return fail(h, REGMEM_ERR_ARG, "null pointer");
  RM_CUDA(h, cudaMemcpyAsync(dst, lse_of(h, h->lse_layer), (size_t)h->heads * h->N * sizeof(float),
                             cudaMemcpyDeviceToDevice, h->stream));
  return REGMEM_OK;
}

regmem_status regmem_synchronize(regmem_t* h) {
  REGMEM_RANGE;
  if (!h) return REGMEM_ERR_ARG;
  if (h->frame_set) {
    if (cudaSetDevice(h->device) != cudaSuccess)
      return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
    RM_CUDA(h, cudaStreamSynchronize(h->stream));
    if (h->sstream) RM_CUDA(h, cudaStreamSynchronize(h->sstream));
    if (h->cstream) RM_CUDA(h, cudaStreamSynchronize(h->cstream));
    if (h->dstream) RM_CUDA(h, cudaStreamSynchronize(h->dstream));
    RM_CUDA(h, cudaGetLastError());
  }
  return check_device_status(h);
}

regmem_status regmem_debug_set(regmem_t* h, int64_t wait_limit_us, int32_t skip_kv_load) {
  REGMEM_RANGE;
  if (!h || wait_limit_us < 1 || wait_limit_us > 60000000 || skip_kv_load < -1)
    return REGMEM_ERR_ARG;
  h->wait_ns = (unsigned long long)wait_limit_us * 1000ull;
  h->fault_skip_kv = skip_kv_load;
  return REGMEM_OK;
}

regmem_status regmem_profile_enable(regmem_t* h, int32_t time_attention) {
  REGMEM_RANGE;
  if (!h) return REGMEM_ERR_ARG;
  if (h->frame_set) {
    if (cudaSetDevice(h->device) != cudaSuccess)
      return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
    for (size_t i = 0; i < h->ev_busy.size(); ++i)
      if (h->ev_busy[i]) RM_CUDA(h, harvest_pair(h, i));
  }
  h->prof = regmem_profile{};
  h->time_every = time_attention > 0 ? time_attention : 0;
  h->clk_next = 0;
  if (h->frame_set && h->time_every > 0) {  // preset the slots, stream-ordered before the launches
    const size_t bytes = 2 * kClockSlots * sizeof(unsigned long long);
    if (!h->kclock) RM_CUDA(h, cudaMalloc(&h->kclock, bytes));
    h->clk_frame.assign(kClockSlots, 0);
    RM_CUDA(h, cudaMemsetAsync(h->kclock, 0xFF, bytes / 2, h->stream));
    RM_CUDA(h, cudaMemsetAsync(h->kclock + kClockSlots, 0, bytes / 2, h->stream));
  }
  h->attn_launch_no = 0;
  return REGMEM_OK;
}

regmem_status regmem_profile_read(regmem_t* h, regmem_profile* out) {
  REGMEM_RANGE;
  if (!h || !out) return REGMEM_ERR_ARG;
  if (h->frame_set) {
    if (cudaSetDevice(h->device) != cudaSuccess)
      return fail(h, REGMEM_ERR_CUDA, "cannot select device %d", h->device);
    RM_CUDA(h, cudaStreamSynchronize(h->stream));
    for (size_t i = 0; i < h->ev_busy.size(); ++i)
      if (h->ev_busy[i]) RM_CUDA(h, harvest_pair(h, i));
    if (h->kclock && h->clk_next > 0) {
      const size_t n = (size_t)h->clk_next;
      std::vector<unsigned long long> t0(n), t1(n);
      RM_CUDA(h, cudaMemcpy(t0.data(), h->kclock, n * sizeof(unsigned long long),
                            cudaMemcpyDeviceToHost));
      RM_CUDA(h, cudaMemcpy(t1.data(), h->kclock + kClockSlots, n * sizeof(unsigned long long),
                            cudaMemcpyDeviceToHost));
      double ns[2] = {0.0, 0.0};
      long long cnt[2] = {0, 0};
      for (size_t i = 0; i < n; ++i) {
        const int f = h->clk_frame[i];
        ++cnt[f];
        if (t1[i] > t0[i]) ns[f] += (double)(t1[i] - t0[i]);
      }
      h->prof.attention_clocked = cnt[0];
      h->prof.attention_clock_ms = ns[0] * 1e-6;
      h->prof.frame_attention_clocked = cnt[1];
      h->prof.frame_attention_clock_ms = ns[1] * 1e-6;
    }
  }
  *out = h->prof;
  return check_device_status(h);
}

void regmem_destroy(regmem_t* h) {
  if (!h) return;
  if (h->frame_set) {
    cudaSetDevice(h->device);
    cudaStreamSynchronize(h->stream);
    if (h->sstream) cudaStreamSynchronize(h->sstream);
    if (h->cstream) cudaStreamSynchronize(h->cstream);
    if (h->dstream) cudaStreamSynchronize(h->dstream);
  }
  cudaFree(h->bankK);
  cudaFree(h->bankV);
  cudaFree(h->lse);
  cudaFree(h->qidx);
  cudaFree(h->part_o);
  cudaFree(h->part_lse);
  cudaFree(h->head_done);
  cudaFree(h->kclock);
  cudaFree(h->adm_lists);
  if (h->status_host) cudaFreeHost(h->status_host);
  cudaFree(h->stQ);
  cudaFree(h->stOut);
  cudaFree(h->stSal);
  for (auto* p : h->stK) cudaFree(p);
  for (auto* p : h->stV) cudaFree(p);
  for (auto e : h->ev_ring) cudaEventDestroy(e);
  for (auto& hs : h->hs) {
    cudaFree(hs.q);
    cudaFree(hs.k);
    cudaFree(hs.v);
    cudaFree(hs.out);
    cudaFree(hs.sal);
    if (hs.h2d) cudaEventDestroy(hs.h2d);
    if (hs.done) cudaEventDestroy(hs.done);
    if (hs.d2h) cudaEventDestroy(hs.d2h);
  }
  if (h->cstream) cudaStreamDestroy(h->cstream);
  if (h->dstream) cudaStreamDestroy(h->dstream);
  if (h->sstream) cudaStreamDestroy(h->sstream);
  if (h->main_ev) cudaEventDestroy(h->main_ev);
  if (h->side_ev) cudaEventDestroy(h->side_ev);
  delete h;
}

}  // extern "C"
