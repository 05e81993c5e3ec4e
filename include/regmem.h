/*
 * regmem.h -- C ABI of the GB300 regulated streaming-attention library
 * (libregmem.so).
 *
 * The library implements the per-frame, per-layer hot path of RegVGGT's
 * streaming inference (arxiv 2609.23286):
 *
 *   1. temporal causal attention of the frame's queries over
 *      [regulated KV memory ; the frame's own keys/values]      (Eq. 2, Eq. 3)
 *   2. LSE-Saliency: per-key attention mass of a sampled query subset,
 *      recovered from the rows' log-sum-exp                      (Sec. 3.3,
 *      "FlashAttention-Compatible Saliency Estimation" and "Head-Specific
 *      Token Retention")
 *   3. per-head top-k admission of the most salient tokens into an append-only
 *      HBM memory; the first frame is stored whole                (Eq. 4, Eq. 6)
 *
 * Conventions for every call
 * --------------------------
 * - Tensors named Q, K, V, out are bfloat16, row-major [N][H][64] (token,
 *   head, channel), i.e. the usual [tokens, heads*head_dim] activation layout;
 *   they are DEVICE pointers owned by the caller, 16-byte aligned.
 * - Work is enqueued asynchronously on the stream given to
 *   regmem_set_stream (default: the legacy default stream).  A call returns
 *   before the GPU has finished.
 * - Every call validates its arguments and the handle's state before
 *   enqueueing anything: on any error it enqueues nothing, changes no state,
 *   returns a negative regmem_status, and regmem_last_error() describes why.
 *   Errors reported by the CUDA runtime are returned as REGMEM_ERR_CUDA.
 *   Device-side bounded waits that expire are reported as REGMEM_ERR_TIMEOUT
 *   by the next call (and by regmem_synchronize); the handle must then be
 *   destroyed.
 * - A handle is not thread-safe: one host thread at a time.
 */
#ifndef REGMEM_H
#define REGMEM_H

#include <stdint.h>

#if defined(__GNUC__)
#define REGMEM_API __attribute__((visibility("default")))
#else
#define REGMEM_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef struct regmem regmem_t; /* opaque; owns the per-layer HBM banks */

typedef enum regmem_status {
  REGMEM_OK = 0,
  REGMEM_ERR_ARG = -1,         /* bad pointer, size, index or value          */
  REGMEM_ERR_STATE = -2,       /* call out of order for the layer's state   */
  REGMEM_ERR_CAPACITY = -3,    /* admission would overflow the bank          */
  REGMEM_ERR_CUDA = -4,        /* CUDA runtime / driver error                */
  REGMEM_ERR_UNSUPPORTED = -5, /* shape outside what the kernels handle      */
  REGMEM_ERR_TIMEOUT = -6,     /* a device-side bounded wait expired         */
  REGMEM_ERR_DEVICE_CHECK = -7 /* a range guard of the checked build failed:
                                  libregmem_checked.so, compiled with
                                  REGMEM_DEVICE_CHECKS, checks the indices its
                                  kernels derive before global accesses      */
} regmem_status;

/* Frame geometry.  Tokens of a frame are ordered [special tokens, patch tokens
 * row-major over a grid_h x grid_w grid]; n_tokens = n_special + grid_h*grid_w
 * (VGGT: 1 camera + 4 register tokens, then 37x37 patches of a 518x518 image
 * at patch 14). */
typedef struct regmem_frame_desc {
  int32_t n_tokens;   /* N, tokens per frame (queries and keys of the frame)     */
  int32_t n_special;  /* leading non-patch tokens                               */
  int32_t grid_h;     /* patch rows                                             */
  int32_t grid_w;     /* patch columns                                          */
  int32_t ds;         /* query down-sampling window (Sec. 3.3: 2 = 2x2); 0 -> 2  */
  int32_t max_frames; /* frames the banks must hold: capacity =
                         N + (max_frames - 1) * budget rows per head and layer */
  float scale;        /* softmax scale; 0 -> 1/sqrt(head_dim) (Eq. 2)            */
  int32_t candidates; /* 0: only patch tokens may be admitted; 1: all tokens      */
} regmem_frame_desc;

/* Creates a handle for `layers` global-attention layers with `heads` heads of
 * `head_dim` channels (head_dim must be 64), admitting at most `budget` rows
 * per head per frame (Eq. 6: k = floor(gamma N); budget >= 0).  Allocates
 * nothing on the GPU yet.  *out receives the handle (NULL on error). */
REGMEM_API regmem_status regmem_create(regmem_t** out, int32_t layers, int32_t heads, int32_t head_dim,
                            int32_t budget);

/* Fixes the frame geometry and allocates, on the current CUDA device, the
 * banks ([layers][heads][capacity][64] bf16 for K and for V, zero-filled),
 * the library's scratch, and the staging buffers, copy streams and events of
 * the host-buffer entry points (six sets of Q, K, V, out and saliency for
 * regmem_attend_admit_host; Q, out, saliency and per-layer K and V for
 * regmem_attend_frame_host: 11.3 MB x 6 + 8.5 MB + 5.6 MB x layers at
 * N = 1374, 16 heads), so that no later call allocates device memory
 * (regmem_profile_enable's launch clock excepted, see there).  Must be
 * called once, before the first attend;
 * ERR_STATE if called again. ERR_UNSUPPORTED if N exceeds 65536 or the
 * number of admission candidates exceeds 8192. */
REGMEM_API regmem_status regmem_set_frame(regmem_t* h, const regmem_frame_desc* fd);

/* Stream (a cudaStream_t passed as void*) on which all later work is
 * enqueued.  NULL selects the legacy default stream. */
REGMEM_API regmem_status regmem_set_stream(regmem_t* h, void* stream);

/* on = 1: regmem_attend_admit (and its host-buffer form) runs the saliency
 * and the admission on a side stream of the handle's own, created at the
 * lowest stream priority, after the call's attention (an event), so that
 * they overlap the next layer's attention instead of following it on the
 * stream.  The attention output `out` is complete in stream order as usual;
 * `saliency`, `idx_out` and the bank update are complete after
 * regmem_synchronize, and Q/K/V must stay valid until then.  The next
 * attend of the same layer is ordered after that layer's side work (the
 * stream waits on an event; one wait covers all side work so far).  For the
 * attention's CTAs to go ahead of the side blocks when both wait for SMs,
 * the stream of regmem_set_stream should have a higher priority than the
 * lowest.  on = 0 (the default) runs everything on the stream; switching it
 * off orders the stream after the pending side work.  The two-call path
 * (regmem_attend_frame + regmem_admit), regmem_export_bank,
 * regmem_import_bank and regmem_reset order the stream after the pending
 * side work first.  ERR_ARG unless on is 0 or 1. */
REGMEM_API regmem_status regmem_set_overlap(regmem_t* h, int32_t on);

/* Orders the stream after all side work enqueued so far (an event wait on
 * the stream; the host does not block), so that work the caller enqueues
 * next on the stream sees the saliency, indices and banks of every earlier
 * call.  Nothing to do without overlap. */
REGMEM_API regmem_status regmem_join(regmem_t* h);

/* Eq. 3 for one layer and the current frame, fused with LSE-Saliency.
 *   out[n][h][:] = softmax(Q_h K_h^T * scale) V_h over the keys
 *                  [bank rows of (layer, h) ; the frame's N keys]
 *   saliency[h][j] = sum over sampled queries i of exp(Z_ij - LSE_i),
 *                  j in [0, N): the frame's keys; LSE_i is taken over every
 *                  attended key, so saliency is the exact full-context
 *                  attention mass (not renormalised over the frame).
 * Q, K, V: device bf16 [N][H][64]; out: device bf16 [N][H][64];
 * saliency: device fp32 [H][N].
 * State: the layer must not have an attend pending (ERR_STATE).  K, V and
 * saliency must stay valid and unmodified, in stream order, until this
 * layer's regmem_admit has been enqueued; the library keeps the pointers. */
REGMEM_API regmem_status regmem_attend_frame(regmem_t* h, int32_t layer, const void* Q, const void* K,
                                  const void* V, void* out, float* saliency);

/* Same as regmem_attend_frame but with HOST buffers: Q, K, V and out are
 * bf16 [N][H][64] and saliency fp32 [H][N] in host memory (pinned for
 * asynchronous copies; pageable also works, synchronously).  K and V are
 * staged into library-owned device buffers (made by regmem_set_frame) that
 * stay valid until admit.
 * The device->host copies of out and saliency are enqueued on the stream:
 * they are complete after regmem_synchronize (or a sync of the stream). */
REGMEM_API regmem_status regmem_attend_frame_host(regmem_t* h, int32_t layer, const void* hostQ,
                                       const void* hostK, const void* hostV, void* hostOut,
                                       float* hostSaliency);

/* Eq. 4 / Eq. 6 for one layer, after its attend.
 * - If the layer's memory is empty, the frame's N rows (all heads) become the
 *   global anchor (Eq. 4) and k is ignored.
 * - Otherwise, per head, the k candidate tokens with the largest saliency
 *   (ties -> lower token index) are appended to that head's bank in ascending
 *   token order (Eq. 6).  0 <= k <= min(budget, candidates) or ERR_ARG;
 *   ERR_CAPACITY if the bank would overflow (nothing is appended).
 * idx_out: optional device int32 [H][k] receiving the admitted token indices
 * (ascending per head); NULL to skip.  On the anchor frame nothing is written.
 * k equal to the number of candidates admits the whole frame (with
 * candidates = 1 and budget >= N: the unregulated full-KV stream, every
 * frame's N rows kept); that case is a plain copy, nothing is ranked.
 * State: the layer must have an attend pending (ERR_STATE). */
REGMEM_API regmem_status regmem_admit(regmem_t* h, int32_t layer, int32_t k, int32_t* idx_out);

/* Admission without head-specific retention (the ablation of Sec. 4.5,
 * Table 4, "w/o Head-specific Retention"): instead of each head ranking its
 * own saliency, one set of k candidate tokens is chosen for all heads, ranked
 * by the saliency summed over heads (fp32, heads added in ascending order;
 * the same order as the head mean), ties -> lower token index, and the rows
 * of those tokens are appended to every head's bank in ascending token order.
 * idx_out: optional device int32 [k].  Everything else (anchor frame, k
 * range, capacity, state) as in regmem_admit. */
REGMEM_API regmem_status regmem_admit_shared(regmem_t* h, int32_t layer, int32_t k, int32_t* idx_out);

/* regmem_attend_frame followed by regmem_admit(layer, k, idx_out), in one
 * call: the whole per-frame step of one layer (Eq. 3, the LSE-Saliency of
 * Sec. 3.3, then Eq. 4 or Eq. 6).  For k <= 32 the admission runs inside the
 * saliency kernel (each key tile keeps its best candidates, the last block of
 * each head merges them and appends), so it needs no launch of its own;
 * larger k takes a separate selection kernel.  Arguments, layouts, k range
 * and errors as in the two
 * calls; every check (including k and capacity) is made before anything is
 * enqueued.  The library keeps no pointer after the call: K, V and saliency
 * need only stay valid until the enqueued work has run (with overlap, that
 * includes the side stream's saliency and admission: regmem_synchronize or
 * regmem_join).
 * State: the layer must not have an attend pending (ERR_STATE); afterwards
 * it has none. */
REGMEM_API regmem_status regmem_attend_admit(regmem_t* h, int32_t layer, const void* Q, const void* K,
                                  const void* V, void* out, float* saliency, int32_t k,
                                  int32_t* idx_out);

/* regmem_attend_frame followed by regmem_admit_shared(layer, k, idx_out), in
 * one call: the per-frame step of one layer with the selection that keeps no
 * head-specific retention (Table 4, first row).  For k <= 32 the selection
 * runs inside the saliency kernel: the last head to finish a key tile ranks
 * the tile's head-summed saliency, and the last tile merges the lists and
 * appends.  Larger k takes the separate selection kernel.  Both run on the
 * stream regmem_attend_admit uses for its side work (the side stream when
 * overlap is on).  Results are bit-identical to the two calls; idx_out is an
 * optional device int32 [k].  Arguments, checks, state and validity of K, V
 * and saliency as in regmem_attend_admit. */
REGMEM_API regmem_status regmem_attend_admit_shared(regmem_t* h, int32_t layer, const void* Q,
                                         const void* K, const void* V, void* out,
                                         float* saliency, int32_t k, int32_t* idx_out);

/* regmem_attend_admit with HOST buffers (layouts as in
 * regmem_attend_frame_host; no index output).  Six library-owned staging
 * sets are used in turn and the copies run on two copy streams of the
 * handle's own (one each way), ordered against the kernels by events: a
 * call's host->device copies overlap the previous call's kernels and its
 * device->host copies the next call's.  Host buffers should be pinned (pageable ones are copied
 * synchronously by CUDA).  The caller must not modify hostQ/hostK/hostV, nor
 * read hostOut/hostSaliency, before regmem_synchronize (which waits for all
 * of the handle's streams); consecutive calls may reuse the same buffers. */
REGMEM_API regmem_status regmem_attend_admit_host(regmem_t* h, int32_t layer, const void* hostQ,
                                       const void* hostK, const void* hostV, void* hostOut,
                                       float* hostSaliency, int32_t k);

/* Non-causal attention inside one frame (the frame-attention layers that
 * alternate with the global ones, Sec. 3.1): out = softmax(Q K^T scale) V
 * over the frame's own N keys, no memory, no saliency.  Uses the geometry of
 * regmem_set_frame.  Layouts as in regmem_attend_frame. */
REGMEM_API regmem_status regmem_frame_attention(regmem_t* h, const void* Q, const void* K, const void* V,
                                     void* out);

/* Empties every layer's memory (length 0, no attend pending); allocations
 * and stream are kept.  Enqueues nothing. */
REGMEM_API regmem_status regmem_reset(regmem_t* h);

/* Rows currently held per head in `layer`'s bank (|M_t| of Eq. 6). */
REGMEM_API regmem_status regmem_memory_len(const regmem_t* h, int32_t layer, int64_t* len);

/* Rows each head's bank can hold (set by regmem_set_frame). */
REGMEM_API regmem_status regmem_capacity(const regmem_t* h, int64_t* rows);

/* Copies `layer`'s bank to host memory: hostK and hostV receive
 * [H][len][64] bf16 with len = regmem_memory_len.  Synchronises the stream. */
REGMEM_API regmem_status regmem_export_bank(regmem_t* h, int32_t layer, void* hostK, void* hostV);

/* Replaces `layer`'s bank with host data [H][len][64] bf16 (checkpoint
 * resume, or teacher forcing in tests).  len <= capacity; clears any pending
 * attend.  Synchronises the stream. */
REGMEM_API regmem_status regmem_import_bank(regmem_t* h, int32_t layer, const void* hostK,
                                 const void* hostV, int64_t len);

/* Enqueues a copy of the LSE rows of the most recent attend (any layer):
 * dst is device fp32 [H][N] (natural log).  Each layer keeps its own LSE
 * rows ([layers][H][N] fp32 of scratch), so the side work of one layer can
 * still read them while the next layer's attention runs. */
REGMEM_API regmem_status regmem_copy_lse(regmem_t* h, float* dst);

/* Waits for all work enqueued on the handle's stream and on its own side and
 * copy streams, and reports any device status (REGMEM_ERR_TIMEOUT) or CUDA
 * error. */
REGMEM_API regmem_status regmem_synchronize(regmem_t* h);

/* Allocation-free attend step.  The paper has no counterpart: this entry
 * point exists for callers that cannot allocate device memory when they run
 * the attention -- code living inside another framework's memory pool or
 * arena, plugins handed pre-sized buffers, real-time loops in which a
 * cudaMalloc could stall on the driver.  It computes what
 * regmem_attend_frame computes (attention over [bank rows ; frame] and the
 * LSE-saliency of the frame's keys) with the same kernels, but needs no
 * handle and allocates nothing: no cudaMalloc, no cudaFree, no allocating
 * library routine.
 *
 * Arguments: fd gives the frame geometry (n_tokens, n_special, grid_h,
 * grid_w, ds, scale; max_frames and candidates are ignored); Q, K, V, out are
 * device bf16 [N][heads][64]; bankK/bankV are the caller's device bank of one
 * layer, bf16 [heads][bank_rows][64], of which the first M rows per head are
 * attended (NULL allowed when M == 0); saliency is device fp32 [heads][N];
 * status is a REQUIRED device (or mapped host) int32 into which the kernels
 * OR nonzero bits if a bounded device-side wait expires; the caller zeroes it
 * before the call and reads it after synchronising, and treats out and
 * saliency as undefined when it is nonzero (there is no handle, so no later
 * call could report the failure; NULL gives REGMEM_ERR_ARG); stream is a
 * cudaStream_t (NULL: legacy default stream).
 * All pointers 16-byte aligned (status 4-byte aligned).
 *
 * Scratch: the kernels' split partials, LSE rows and sampled-query list live
 * in one file-scope device array of 11.9 MB that every GPU which loads this
 * library holds until the process exits.  Limits, rejected with
 * REGMEM_ERR_UNSUPPORTED before anything is enqueued: heads * N <= 262144,
 * N <= 65536, sampled queries <= 8192, and the attention grid (one CTA per
 * SM) <= 160 CTAs.  Bad arguments give REGMEM_ERR_ARG; there is no handle, so no
 * error message is kept.
 * Every call on a device shares that one array and leaves its contents
 * behind; calls whose work overlaps on the GPU (two streams, or two host
 * threads) race on it, so serialise them.  The first call on each device,
 * with that device current, looks up the array's device address and sets
 * kernel attributes; make that first call before any stream capture. */
REGMEM_API regmem_status regmem_attend_frame_noalloc(const regmem_frame_desc* fd, int32_t heads,
                                                     const void* Q, const void* K, const void* V,
                                                     const void* bankK, const void* bankV,
                                                     int64_t bank_rows, int64_t M, void* out,
                                                     float* saliency, int32_t* status,
                                                     void* stream);

/* Failure-detection hook, for tests.  The paper has no counterpart.
 * wait_limit_us sets the limit of every bounded wait inside the attention
 * kernel for this handle's later launches (default 2,000,000 us = 2 s;
 * 1 <= wait_limit_us <= 60 s).  skip_kv_load >= 0 arms a one-shot fault for
 * the NEXT attention launch only: the first CTA's TMA producer does not
 * issue its skip_kv_load-th K/V tile load (CTA-local index, from 0), so
 * nothing ever lands in that ring stage; the consumers' bounded waits on it
 * run out after the limit, every role of that CTA stops, drains the copies
 * and MMAs it has issued, frees its tensor memory and sets the timeout bit
 * of the handle's status word.  The GPU context stays usable: the next call
 * (and regmem_synchronize) returns REGMEM_ERR_TIMEOUT and the handle must
 * then be destroyed.  The index must be below the number of K/V loads of the
 * first CTA, else nothing is skipped.  skip_kv_load = -1 disarms.  Nothing
 * is enqueued.  ERR_ARG on out-of-range values. */
REGMEM_API regmem_status regmem_debug_set(regmem_t* h, int64_t wait_limit_us, int32_t skip_kv_load);

/* Launch counters and kernel timing, for measurement tools.
 * Counters cover every kernel this handle launched since the last
 * regmem_profile_enable.  When time_attention is set, CUDA events are
 * recorded on the handle's stream immediately before and after the sampled
 * launches of the attention kernel and after the merge of split units that
 * follows it: attention_ms sums the attention kernel's intervals, merge_ms
 * the merge's; the other kernels are not bracketed.  It also turns on the
 * attention kernel's own launch clock for EVERY attention launch: the GPU's
 * global timer from the first CTA past the launch's dependency wait to the
 * last CTA's end, kept per launch in 16 MB of device memory (allocated by
 * the first regmem_profile_enable after regmem_set_frame) for up to 2^20
 * launches per profiling window, and summed by regmem_profile_read.  No
 * event sits between launches, so it does not perturb the stream it
 * measures. */
typedef struct regmem_profile {
  int64_t launches_attention; /* attention kernel (attend and frame attention)  */
  int64_t launches_saliency;  /* LSE-saliency kernel                            */
  int64_t launches_admit;     /* top-k + append kernel                          */
  int64_t launches_anchor;    /* first-frame copy kernel                        */
  int64_t launches_combine;   /* merge of units split between attention CTAs   */
  int64_t attention_timed;    /* attention launches with an event pair          */
  double attention_ms;        /* summed event time of those launches (the
                                 attention kernel alone)                        */
  double attention_flops;     /* algorithmic 4*N*(M+N)*64*H of those launches   */
  double attention_bytes;     /* algorithmic HBM bytes of those launches:
                                 Q, O, K/V of the attended rows, LSE           */
  int32_t attention_ctas;     /* grid of the most recent attention launch      */
  int32_t attention_ctas_per_sm; /* resident attention CTAs per SM (occupancy) */
  double merge_ms;            /* summed event time of the merges of split units
                                 behind those launches                          */
  int64_t attention_clocked;  /* regulated attention launches (attend calls)
                                 measured by the launch clock                   */
  double attention_clock_ms;  /* their summed durations (global timer)          */
  double attention_clock_flops; /* algorithmic FLOPs of those launches          */
  int64_t launches_frame_attention; /* of launches_attention: regmem_frame_attention */
  int64_t frame_attention_clocked;  /* frame-attention launches measured by the
                                       launch clock                              */
  double frame_attention_clock_ms;  /* their summed durations                   */
  double frame_attention_clock_flops; /* their algorithmic FLOPs, 4 N^2 64 H each */
} regmem_profile;

/* Resets the counters; time_attention = n >= 1 also brackets every n-th
 * attention launch with events (0 stops it).  Kernels are launched so that
 * each may start while its predecessor in the stream finishes; an event pair
 * between two launches removes that overlap at those two boundaries, so a
 * sparse sample (n of 8 or more) perturbs a long run least. */
REGMEM_API regmem_status regmem_profile_enable(regmem_t* h, int32_t time_attention);

/* Waits for the handle's stream and fills *out. */
REGMEM_API regmem_status regmem_profile_read(regmem_t* h, regmem_profile* out);

/* Human-readable description of the last error on this handle ("" if none). */
REGMEM_API const char* regmem_last_error(const regmem_t* h);

/* Name of a status code. */
REGMEM_API const char* regmem_status_string(regmem_status s);

/* Frees every allocation of the handle (waits for its stream first). */
REGMEM_API void regmem_destroy(regmem_t* h);

#ifdef __cplusplus
}
#endif

#endif /* REGMEM_H */
