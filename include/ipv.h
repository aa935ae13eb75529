/*
 * ipv.h -- C ABI of the GB300 (sm_103a) InfiniPot-V KV-cache compression pass.
 *
 * InfiniPot-V (arXiv 2506.15745) keeps a streaming video MLLM's KV cache under
 * a fixed memory cap |M|: whenever the cache reaches |M| tokens it is cut to a
 * target size |C| (Algorithm 1). For every (layer, KV head) "slab" the pass
 *   (i)   scores each past vision token with Temporal-axis Redundancy
 *         s_TaR = -(1/r) sum_{t'} cos(K_past[t,i,j], K_recent[t',i,j])
 *         (Sec. 3.1, Eq. tar; the cache is viewed as f frames of p patches,
 *         the r latest frames are "recent");
 *   (ii)  scores it with Value Norm s_VaN = ||V[t,i,j]||_2 (Sec. 3.2);
 *   (iii) keeps the r*p recent tokens, then the floor(alpha |C|) - r*p past
 *         tokens of highest s_TaR, then fills the rest of |C| with the past
 *         tokens of highest s_VaN that TaR did not take (Sec. 3.3, Algorithm 1
 *         steps 3-5; Algorithm 2's max-forcing of TaR picks before its final
 *         TopK); ties go to the lower token index, NaN ranks lowest;
 *   (iv)  compacts K and V to the kept rows in ascending index order
 *         (Sec. 3.1, K~ = K[:, I, :]; Algorithm 2 last step).
 * Optionally (ipv_options.van_pool) step (iii) ranks a layer-adaptive average
 * pooling of VaN instead of raw VaN (Sec. 3.2 "Layer-wise Adaptive Pooling";
 * Algorithm 2): per layer, CV = sigma/mu of VaN over all its heads and cached
 * tokens picks a pool size k = g(CV) in {7, 5, 3, 1}, and a token's pooled
 * VaN is the mean VaN of the cached tokens of its own frame within the k x k
 * window around its grid position (stride 1; positions outside the grid or
 * no longer cached are left out; sigma is the population deviation).
 *
 * Memory layout (all device memory, owned by the caller unless stated):
 *   K or V cache half : [n_layers][n_kv_heads][token_capacity][head_dim],
 *                       contiguous, element type chosen in ipv_init (bf16 or
 *                       fp32), 16-byte aligned; row n of slab s starts at
 *                       element (s * token_capacity + n) * head_dim.
 *   patch ids         : uint16 [n_layers][n_kv_heads][token_capacity]: the
 *                       frame-grid position (i*w + j) of each cached token.
 *   frame ids         : uint32, same layout: the frame each cached token came
 *                       from (only equality matters). Pooled VaN needs them
 *                       once the cache has been compacted.
 *   scores            : fp32 [n_slabs][n_tokens].
 *   kept indices      : int32 [n_slabs][budget], ascending per slab.
 *
 * Frames: the n_tokens rows of a slab hold f = n_tokens / p frames' worth of
 * tokens (p = frame_grid_h * frame_grid_w). The last r*p rows are the r most
 * recent frames, whole and in patch order. The patch of a past row n is
 * patch_id[n] when the cache half has patch ids, else n mod p (a cache that
 * has never been compacted); likewise its frame is frame_id[n], else n div p.
 * With ids, rows are in increasing (frame id, patch id) order, as appending
 * whole frames with increasing frame ids and this pass's in-order compaction
 * keep them (pooled VaN relies on it; no check is made).
 *
 * Execution: every compute entry point validates its arguments on the host,
 * then enqueues kernels on the given CUDA stream and returns without waiting.
 * No entry point synchronises the device or the stream, and none allocates
 * device memory except ipv_init. The library keeps one global state (device,
 * element type, scratch); calls are not thread-safe and must come from one
 * host thread at a time. The scratch (scores, recent-frame means, the
 * compaction's work counters) is shared by every ipv_compress and ipv_score
 * call: two such calls whose kernels could overlap on the GPU (different
 * streams with no event or stream order between them) race on it, so enqueue
 * them on one stream or order them with events. ipv_select, ipv_van_pool and
 * ipv_append_frames touch only the caller's buffers, and host-device copies
 * on other streams may overlap any call. Errors never trap on the device.
 */
#ifndef IPV_H_
#define IPV_H_

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
  IPV_OK = 0,
  IPV_EINVAL = 1,   /* bad argument; nothing was enqueued */
  IPV_ENOINIT = 2,  /* ipv_init has not succeeded (or ipv_shutdown was called) */
  IPV_ENOMEM = 3,   /* device allocation failed in ipv_init */
  IPV_ECUDA = 4,    /* CUDA runtime error; see ipv_last_error() */
  IPV_ETIMEOUT = 5  /* a bounded host wait ran out (profiling read-back only) */
} ipv_status;

typedef enum { IPV_BF16 = 0, IPV_F32 = 1 } ipv_dtype;

typedef struct {
  int device;             /* CUDA device ordinal */
  ipv_dtype dtype;        /* element type of K and V */
  int recent_frames;      /* r; 0 = max(1, floor(f/8 + 1/2)), the r = 0.125 f
                             default of Appendix B.2 */
  int max_head_dim;       /* largest head_dim any call will use (<= 512) */
  int max_frame_tokens;   /* largest p = frame_grid_h*frame_grid_w (<= 65535) */
  int64_t max_slabs;      /* largest n_layers*n_kv_heads any call will use */
  int64_t token_capacity; /* rows per slab in each cache half (the slab stride) */
  int single_kernel;      /* 0: ipv_compress runs the pass as its four step kernels
                             (recent-frame mean, scoring, selection, compaction),
                             one after the other; 1: as one fused persistent kernel
                             (cooperative launch, two blocks per SM) that works
                             through the slabs in order and compacts each slab a few
                             slabs after scoring it, so that its kept rows are read
                             from L2 instead of HBM. The fused kernel takes caches
                             that have never been compacted (the live half has no
                             patch ids) and whose selection keys fit the registers
                             of one block (n_tokens - r*p <= 9216 past tokens);
                             other calls run the step kernels. Both give
                             bit-identical results; the fused kernel is the
                             slower one (a slab's selection outlasts its rows'
                             stay in L2). */
  int van_pool;           /* 0: the VaN stage ranks raw VaN (Sec. 3.2 s_VaN);
                             1: it ranks layer-adaptive pooled VaN (Sec. 3.2,
                             Algorithm 2); needs single_kernel = 0 and
                             max_frame_tokens <= IPV_MAX_POOL_FRAME_TOKENS */
  float cv_tau[3];        /* tau_1 <= tau_2 <= tau_3 (van_pool = 1): pool size
                             g(CV) = 7 if CV < tau_1, 5 if CV < tau_2, 3 if
                             CV < tau_3, else 1 (Algorithm 2; the paper's values
                             are model-specific and unpublished) */
  int head_shared;        /* 0: one index set per (layer, KV head) slab;
                             1: one per layer, shared by its KV heads (Sec. 3.1:
                             K in R^{H x N x D} compressed as K[:, I, :]): a
                             token's key and value are its H x D blocks, TaR
                             uses their l2-normalised (Frobenius) cosine and
                             VaN their norm, kept_idx_out is [n_layers][budget]
                             and every head is compacted with its layer's
                             indices. Needs single_kernel = 0 and
                             n_kv_heads*head_dim*element size <= 2048 bytes. */
  int ablation;           /* IPV_ABLATION_*: a variant of the ablation study
                             (Sec. 4, ablation table) for comparisons; needs
                             single_kernel = 0 */
} ipv_options;

/* Ablation variants (Sec. 4 ablation table). TAR_REVERSE / VAN_REVERSE: the
 * stage keeps the past tokens of lowest TaR / VaN instead of highest (NaN
 * still ranks last, ties still go to the lower index). TAR_FRAME: frame-level
 * redundancy, each past token's TaR replaced by the mean TaR of the cached
 * past tokens of its frame (needs frame ids once the cache holds patch ids,
 * and frame_grid_h*frame_grid_w <= IPV_MAX_POOL_FRAME_TOKENS). UNIFORM:
 * "Uniform Select" (Sec. 4, KV cache compression details: frames at regular
 * intervals, all their tokens kept), which reads no score: the n_tokens rows
 * are F = n_tokens/p frames of p consecutive rows, and the pass keeps the
 * k = budget/p whole frames F - 1 - floor(i F / k), i = 0..k-1 (every
 * (F/k)-th frame counting back from the newest), in ascending row order.
 * budget must be a multiple of p (else IPV_EINVAL); the recent-frame rule
 * r*p < budget does not apply. Compacting whole frames keeps the cache whole
 * frames, so a stream compressed this way stays in the frame view. */
enum {
  IPV_ABLATION_NONE = 0,
  IPV_ABLATION_TAR_REVERSE = 1,
  IPV_ABLATION_VAN_REVERSE = 2,
  IPV_ABLATION_TAR_FRAME = 3,
  IPV_ABLATION_UNIFORM = 4
};

/* One tensor (K or V) of the ping-pong cache: two halves of identical
 * layout; buf[cur] holds the live rows. patch_id[h] and frame_id[h] may be
 * NULL. */
typedef struct {
  void* buf[2];
  uint16_t* patch_id[2];
  int cur;
  uint32_t* frame_id[2];
} ipv_kv;

/* Largest n_tokens the selection kernel accepts (its keys live in shared memory). */
#define IPV_MAX_TOKENS 49152
/* Largest frame (frame_grid_h*frame_grid_w) pooled VaN accepts; the grid
 * must also satisfy (frame_grid_h + 6) * (frame_grid_w + 6) <= 14080 (a
 * frame's VaN map, with a 3-cell border, is held in shared memory per warp). */
#define IPV_MAX_POOL_FRAME_TOKENS 4096

/* Initialise the library on opt->device: checks the device, allocates the
 * scratch (per-token scores and per-patch recent-frame means, sized from
 * max_slabs, token_capacity, max_frame_tokens and max_head_dim). Calling it
 * again first releases the previous state. Errors: IPV_EINVAL (bad options),
 * IPV_ECUDA (no usable device), IPV_ENOMEM. */
ipv_status ipv_init(const ipv_options* opt);

/* Release the scratch and forget the options. Waits for the device first. */
void ipv_shutdown(void);

/* The compression pass, steps (i)-(iv) above, for every (layer, KV head) slab.
 *   k, v          : caches; rows 0..n_tokens-1 of buf[cur] are read, the
 *                   budget survivors are written to rows 0..budget-1 of
 *                   buf[1-cur] and cur is flipped (host-side) in both structs.
 *                   Patch ids: read from k->patch_id[k->cur] (NULL: n mod p);
 *                   written to k->patch_id[1-k->cur] if it is not NULL.
 *                   Frame ids likewise (k->frame_id; NULL: n div p); with
 *                   van_pool a cache with patch ids must have frame ids.
 *                   v->patch_id and v->frame_id are not used.
 *   n_tokens      : |M|, rows currently cached per slab; multiple of p.
 *   budget        : |C|, rows kept per slab; r*p < budget.
 *   tar_ratio     : alpha in [0, 1]; the TaR share is floor(alpha * budget).
 *   kept_idx_out  : device int32 [n_layers*n_kv_heads][budget]: the kept
 *                   source rows, ascending per slab ([n_layers][budget],
 *                   per layer, with head_shared).
 *   stream        : a cudaStream_t (NULL = legacy default stream).
 * Pass-through: if n_tokens <= budget nothing is evicted: kept_idx_out gets
 * 0..n_tokens-1 then -1 padding, no row is copied and cur is not flipped.
 * Errors: IPV_EINVAL (checked before anything is enqueued: non-positive
 * sizes, n_tokens not a multiple of p or above token_capacity or
 * IPV_MAX_TOKENS, budget above token_capacity, tar_ratio outside [0,1] or NaN,
 * r*p >= budget, head_dim*elem_size not a multiple of 16 bytes, sizes above
 * the ipv_init maxima, NULL or misaligned pointers, the two halves aliasing,
 * van_pool with patch ids but no frame ids or a grid too large for pooling),
 * IPV_ENOINIT, IPV_ECUDA (launch failure). */
ipv_status ipv_compress(ipv_kv* k, ipv_kv* v, int n_layers, int n_kv_heads, int head_dim,
                        int64_t n_tokens, int frame_grid_h, int frame_grid_w, int64_t budget,
                        float tar_ratio, int32_t* kept_idx_out, void* stream);

/* Steps (i) and (ii) only, for inspection and parity checks: fp32 s_TaR and
 * s_VaN of every token of every slab into tar_out / van_out (device,
 * [n_slabs][n_tokens]; [n_layers][n_tokens] of per-layer scores with
 * head_shared; with the TAR_FRAME ablation tar_out holds the frame means the
 * selection ranks). Entries of the r recent frames are written as 0,
 * except that with van_pool van_out holds the VaN of recent rows too (the
 * layer's CV counts every cached token). Requires n_tokens > r*p. Same
 * argument rules as ipv_compress (budget and tar_ratio aside); the caches are
 * only read. */
ipv_status ipv_score(const ipv_kv* k, const ipv_kv* v, int n_layers, int n_kv_heads,
                     int head_dim, int64_t n_tokens, int frame_grid_h, int frame_grid_w,
                     float* tar_out, float* van_out, void* stream);

/* Step (iii) only: the split-budget selection on given fp32 scores (device,
 * [n_slabs][n_tokens]; entries of the recent frames are ignored), writing
 * kept_idx_out as ipv_compress does. Pass-through and errors as ipv_compress. */
ipv_status ipv_select(const float* tar, const float* van, int64_t n_slabs, int64_t n_tokens,
                      int frame_grid_h, int frame_grid_w, int64_t budget, float tar_ratio,
                      int32_t* kept_idx_out, void* stream);

/* The pooling of VaN alone (Sec. 3.2 "Layer-wise Adaptive Pooling";
 * Algorithm 2 CV, g and AveragePool2d steps), for inspection and parity
 * checks; the pass runs the same kernel. Works for either van_pool setting.
 *   van          : device fp32 [n_layers*n_kv_heads][n_tokens]: VaN of every
 *                  cached row (norms: non-negative or NaN); slabs
 *                  l*n_kv_heads .. l*n_kv_heads + n_kv_heads-1 form layer l.
 *   patch_id, frame_id : device [n_slabs][id_stride] uint16 / uint32, both
 *                  NULL (row n is patch n mod p of frame n div p) or both set,
 *                  rows in increasing (frame, patch) order.
 *   cv_tau       : host, the three thresholds (tau_1 <= tau_2 <= tau_3).
 *   pooled_out   : device fp32 [n_slabs][n_tokens], every row written; a row
 *                  whose patch id is >= p gets NaN when k > 1.
 *   pool_size_out: device int32 [n_layers] (may be NULL): k of each layer.
 * CV is computed in fp32 (two passes: mean, then squared deviations).
 * Errors: IPV_EINVAL (non-positive sizes, n_tokens above IPV_MAX_TOKENS,
 * p above IPV_MAX_POOL_FRAME_TOKENS or a grid too large for its bordered map,
 * id_stride < n_tokens, only one id array,
 * unordered or NaN thresholds, NULL or misaligned pointers), IPV_ENOINIT,
 * IPV_ECUDA. */
ipv_status ipv_van_pool(const float* van, const uint16_t* patch_id, const uint32_t* frame_id,
                        int64_t id_stride, int n_layers, int n_kv_heads, int64_t n_tokens,
                        int frame_grid_h, int frame_grid_w, const float cv_tau[3],
                        float* pooled_out, int32_t* pool_size_out, void* stream);

/* Algorithm 1's accumulate step ("accumulate KV embeddings until reaching
 * |M|") for a streaming cache: appends n_new_frames whole frames behind the
 * rows already cached, in every slab of the live halves buf[cur].
 *   k_new, v_new : device [n_layers*n_kv_heads][n_new_frames*p][head_dim],
 *                  contiguous, the element type of ipv_init (the model's K and
 *                  V of the new frames, patch-major within a frame).
 *   row0         : rows already cached per slab; the new rows go to row0 ..
 *                  row0 + n_new_frames*p - 1 (row0 + those <= token_capacity).
 *   Patch ids (if k->patch_id[cur]): the frame-grid position, (row - row0)
 *   mod p. Frame ids (if k->frame_id[cur]): the frame id of row row0-1 plus
 *   1, 2, ... per new frame, or first_frame, first_frame + 1, ... when row0
 *   is 0; numbered on the device, so a captured CUDA graph that replays
 *   "append, then ipv_compress" keeps counting frames. Together the two ids
 *   are each row's position metadata: (frame, i, j) for a decoder that
 *   re-applies rotary positions after compression (App. B.4), and the row
 *   order for one that re-indexes positions 0..|M|-1.
 * Enqueued on stream, no allocation, cur is not changed. Errors: IPV_EINVAL
 * (NULL or misaligned pointers, non-positive sizes, rows beyond
 * token_capacity, sizes above the ipv_init maxima), IPV_ENOINIT, IPV_ECUDA. */
ipv_status ipv_append_frames(ipv_kv* k, ipv_kv* v, const void* k_new, const void* v_new, int n_layers,
                             int n_kv_heads, int head_dim, int64_t row0, int n_new_frames,
                             int frame_grid_h, int frame_grid_w, uint32_t first_frame, void* stream);

/* The recent-frame count r the library uses for a cache of n_frames frames
 * (the ipv_init override if set, else max(1, floor(n_frames/8 + 1/2))).
 * Returns -1 before ipv_init. */
int ipv_recent_frames(int64_t n_frames);

/* Message of the last failed call on this thread ("" if none). */
const char* ipv_last_error(void);

/* Static name of a status code. */
const char* ipv_status_string(ipv_status s);

/* Kernel timing for benchmarks: while enabled, ipv_compress and ipv_score
 * record CUDA events around each kernel on the call's stream. Kernel ids:
 * 0 recent-frame mean, 1 scoring, 2 selection, 3 compaction, 4 the
 * fused pass (single_kernel = 1), 5 VaN pooling, 6 the per-layer combination of head
 * sums (head_shared). The frame-level TaR kernel of the TAR_FRAME ablation
 * is not timed. */
#define IPV_NUM_KERNELS 7
ipv_status ipv_profile_enable(int on);

/* Waits (at most timeout_ms) for the recorded events, then writes per kernel
 * id the summed device time in ms and the number of launches, and clears the
 * record. Errors: IPV_ETIMEOUT, IPV_ECUDA, IPV_EINVAL (NULL outputs). */
ipv_status ipv_profile_collect(double ms_out[IPV_NUM_KERNELS],
                               int64_t launches_out[IPV_NUM_KERNELS], int timeout_ms);

/* ipv_compress without any device allocation, for callers that cannot
 * allocate device memory: a process whose device memory belongs to a caching
 * allocator or to a fixed budget the library must not grow, or code on a path
 * where cudaMalloc/cudaFree (which can synchronise the device) are not allowed.
 * The paper has no counterpart; this is a deployment variant of the same pass.
 *
 * Same arguments, layout and results as ipv_compress, except that the options
 * of ipv_init (element type, slab stride token_capacity, recent_frames; 0 =
 * default r) are passed in, and no ipv_init is needed. Runs on the current
 * device. The kernels' working memory (TaR and VaN of every token, fp32
 * [n_slabs][n_tokens] each, and the recent-frame mean of every patch, fp32
 * [n_slabs][p][head_dim], each rounded up to 256 bytes) comes from one
 * statically sized array of IPV_STATIC_SCRATCH_BYTES in the library's device
 * image, held on every device that loads the library until the process exits.
 * A pass that needs more is rejected with IPV_EINVAL before anything is
 * enqueued (the LLaVA-OV-7B and Qwen2-VL-7B shapes fit).
 * The first call on a device sets that device up once (kernel limits and
 * cudaGetSymbolAddress of the array): make it before any stream capture. That
 * set-up is kept until the process exits, so resetting the device
 * (cudaDeviceReset) after the first call is not supported. All
 * calls on a device share the array, so calls that may overlap on the GPU
 * race and must be ordered by the caller. Errors: as ipv_compress, plus
 * IPV_EINVAL for a pass too large for the array. */
#define IPV_STATIC_SCRATCH_BYTES (32u << 20)
ipv_status ipv_compress_static(ipv_kv* k, ipv_kv* v, ipv_dtype dtype, int64_t token_capacity,
                               int recent_frames, int n_layers, int n_kv_heads, int head_dim,
                               int64_t n_tokens, int frame_grid_h, int frame_grid_w, int64_t budget,
                               float tar_ratio, int32_t* kept_idx_out, void* stream);

/* Diagnostic: the fused pass (single_kernel = 1) bounds every wait and, when
 * one runs out, sets bits in a device error word (1: a block gave up waiting
 * for its slab's scores before the selection; 2: a block gave up waiting for
 * a slab's selection before compacting it). This waits for the whole device,
 * copies the word to *err_out (0 = no timeout since the last read) and clears
 * it. Errors: IPV_ENOINIT, IPV_EINVAL, IPV_ECUDA. */
ipv_status ipv_device_error(uint32_t* err_out);

/* Diagnostic: the number of polls after which each wait of the fused
 * pass gives up (0 restores the default, 2^20 polls of about 0.1-0.3 us). A
 * wait that gives up sets its bit in the device error word and the pass goes
 * on without the awaited data: its results are then invalid, the device
 * stays usable, and the next pass starts from clean counters. A short
 * limit makes a pass fail fast instead of waiting; tests use it to exercise
 * the error path. Takes effect at the next ipv_compress. Errors:
 * IPV_EINVAL (negative), IPV_ENOINIT. */
ipv_status ipv_set_wait_limit(int64_t polls);

#ifdef __cplusplus
}
#endif

#endif /* IPV_H_ */
