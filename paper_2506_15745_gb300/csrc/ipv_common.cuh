// Internal declarations shared by the kernel translation units of libipv.so.
// Not installed; the public interface is include/ipv.h.
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

namespace ipv {

constexpr float kNormEps = 1e-12f;   // cos(a,b) = a.b / (max|a|,eps)(max|b|,eps)
#ifndef IPV_SELECT_THREADS
#define IPV_SELECT_THREADS 1024
#endif
constexpr int kSelectThreads = IPV_SELECT_THREADS;  // threads of the step path's selection block
#ifndef IPV_SELECT_REG_E
#define IPV_SELECT_REG_E 16
#endif
constexpr int kSelectRegE = IPV_SELECT_REG_E;  // past tokens per thread when the selection keeps its keys in registers
constexpr int kSelectBins = 2048;
constexpr int64_t kMaxTokens = 49152;  // IPV_MAX_TOKENS: selection keys live in shared memory

// ---------------------------------------------------------------- device helpers
// 16-byte global load that bypasses L1 (each cache row is read once per
// kernel). Only for data no thread writes while the kernel runs.
__device__ __forceinline__ uint4 ld_stream(const void* p) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p));
  return r;
}

// L2 eviction policies (createpolicy) for the loads below: a scan that is
// read once marks its lines evict-first, so that lines read earlier and
// wanted again later in the pass (marked evict-last) stay in L2.
__device__ __forceinline__ uint64_t l2_evict_first() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(p));
  return p;
}
__device__ __forceinline__ uint64_t l2_evict_last() {
  uint64_t p;
  asm volatile("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(p));
  return p;
}

// ld_stream with an L2 eviction policy.
__device__ __forceinline__ uint4 ld_stream(const void* p, uint64_t policy) {
  uint4 r;
  asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0,%1,%2,%3}, [%4], %5;"
               : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
               : "l"(p), "l"(policy));
  return r;
}

// 16-byte global store marked evict-first in L2.
__device__ __forceinline__ void st_stream(void* p, uint4 v) {
  asm volatile("st.global.cs.v4.u32 [%0], {%1,%2,%3,%4};" ::"l"(p), "r"(v.x), "r"(v.y), "r"(v.z),
               "r"(v.w)
               : "memory");
}

// ---------------------------------------------------------------- dependent launch
// Programmatic dependent launch: a kernel lets the next kernel of the stream
// start its blocks as soon as every block of this one has started (trigger),
// and a kernel waits for the previous kernel's completion and memory before
// reading its results (wait). Without the launch attribute both are no-ops.
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// Launches kernel on st; with pdl the launch may overlap the previous kernel
// of the stream, which the kernel must then wait for with pdl_wait().
template <typename... Params, typename... Args>
cudaError_t launch(void (*kernel)(Params...), unsigned grid, unsigned block, size_t smem,
                   cudaStream_t st, bool pdl, Args... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(block);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 1 : 0;
  return cudaLaunchKernelEx(&cfg, kernel, args...);
}

// ---------------------------------------------------------------- asynchronous copies
__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

// 16-byte asynchronous copy from global into shared memory through L2 only
// (cp.async.cg); a thread's copies complete at its cp_async_wait_all().
// Both addresses are 16-byte aligned.
__device__ __forceinline__ void cp_async16(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(smem_u32(smem_dst)), "l"(gsrc) : "memory");
}
// Bulk prefetch of [p, p + bytes) into L2; p 16-byte aligned, bytes a multiple of 16.
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
// 4-byte asynchronous copy from global into shared memory (cp.async.ca);
// both addresses 4-byte aligned.
__device__ __forceinline__ void cp_async4(void* smem_dst, const void* gsrc) {
  asm volatile("cp.async.ca.shared.global [%0], [%1], 4;" ::"r"(smem_u32(smem_dst)), "l"(gsrc) : "memory");
}
__device__ __forceinline__ void cp_async_wait_all() { asm volatile("cp.async.wait_all;" ::: "memory"); }

// Elements held by one 16-byte chunk, widened to fp32.
template <typename T>
struct Chunk;

// Elements are handled in consecutive pairs so that sums can use the packed
// fp32 FMA (each lane of fma.rn.f32x2 is an ordinary IEEE fma).
template <>
struct Chunk<uint16_t> {  // bf16 bit patterns
  static constexpr int kElems = 8;
  static constexpr int kPairs = 4;
  __device__ __forceinline__ static void widen2(uint4 c, float2* x) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
#pragma unroll
    for (int i = 0; i < 4; ++i)
      x[i] = make_float2(__uint_as_float(w[i] << 16), __uint_as_float(w[i] & 0xFFFF0000u));
  }
};

template <>
struct Chunk<float> {
  static constexpr int kElems = 4;
  static constexpr int kPairs = 2;
  __device__ __forceinline__ static void widen2(uint4 c, float2* x) {
    x[0] = make_float2(__uint_as_float(c.x), __uint_as_float(c.y));
    x[1] = make_float2(__uint_as_float(c.z), __uint_as_float(c.w));
  }
};

__device__ __forceinline__ float2 fma2(float2 a, float2 b, float2 c) { return __ffma2_rn(a, b, c); }

// Order-preserving 32-bit key of a score: larger float -> larger key; -0 and
// +0 are the same key; every NaN maps to 1, below every number (the smallest
// number, -inf, maps to 0x007FFFFF). Keys 0 and 0xFFFFFFFF are never produced
// and serve as "excluded" / "taken" marks in the selection kernel.
__device__ __forceinline__ uint32_t score_key(float x) {
  if (x != x) return 1u;
  const uint32_t b = __float_as_uint(x + 0.0f);
  return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

// ---------------------------------------------------------------- host launchers
struct ScoreArgs {
  const void* k;            // [S][cap][D]
  const void* v;
  const uint16_t* patch_id; // [S][cap] or nullptr
  int64_t n_slabs, cap, n_tokens;
  int D, p, r;
  int is_bf16;
  float* m;                 // scratch [S][p][D] fp32
  float* tar;               // [S][n_tokens]
  float* van;
  int zero_recent;          // write 0 to the recent-frame entries of tar (and van unless van_recent)
  int van_recent;           // write the VaN of the recent rows to van (pooled VaN's CV counts them)
  int hs;                   // recent-frame mean only: heads per token block (> 1: the shared index
                            // set; slab s is layer s of hs heads, m is written per head-slab)
  float* kk;                // scoring only: if set, write per-head partial sums instead of scores:
                            // tar <- k.m_q, kk <- |k|^2, van <- |v|^2 (NaN without a patch)
  int num_sms;
};

int row_shape(int D, int is_bf16);  // encoded (lanes per row, chunks per lane)
cudaError_t launch_recent_mean(const ScoreArgs& a, cudaStream_t st);
cudaError_t launch_score(const ScoreArgs& a, cudaStream_t st);
size_t score_smem_bytes(int p, int D);
cudaError_t score_prepare(int max_p, int max_D);

struct SelectArgs {
  const float* tar;   // [S][n_tokens]
  const float* van;
  int64_t n_slabs, n_tokens;
  int64_t rp, n_tar, n_van, budget;
  int32_t* kept;      // [S][budget]
  int neg_tar, neg_van;  // ablation: the stage ranks its negated scores (the lowest first)
  int van_smem;       // set by launch_select: VaN is read into shared memory with TaR, up front
  int num_sms;        // > 0: the keys-in-shared-memory selection runs one block per SM, each
                      // looping over slabs (else one block per slab)
};

cudaError_t launch_select(const SelectArgs& a, cudaStream_t st);
cudaError_t launch_passthrough(int32_t* kept, int64_t n_slabs, int64_t n_tokens, int64_t budget,
                               cudaStream_t st);
size_t select_smem_bytes(int64_t n_past);
cudaError_t select_prepare(int64_t max_tokens);
// "Uniform Select" ablation: kept [units][budget] = the rows of the budget/p
// whole frames F - 1 - floor(i F / k) of F = n_tokens/p, ascending.
cudaError_t launch_uniform(int32_t* kept, int64_t units, int64_t n_tokens, int p, int64_t budget,
                           cudaStream_t st);

struct GatherArgs {
  const void* k_src;
  const void* v_src;
  void* k_dst;
  void* v_dst;
  const uint16_t* pid_src;  // nullptr: patch = n mod p
  uint16_t* pid_dst;        // nullptr: not written
  const uint32_t* fid_src;  // nullptr: frame = n div p
  uint32_t* fid_dst;        // nullptr: not written
  const int32_t* kept;      // [S / heads_per_kept][budget]
  int64_t n_slabs, cap, budget;
  int row_bytes, p;
  int num_sms;
  int heads_per_kept;       // head-slabs sharing one row of kept (0 or 1: one each)
  int64_t n_tokens, rp;     // rp > 0: the last rp kept rows of every slab are the rows
                            // n_tokens - rp .. n_tokens - 1 (the recent frames, always kept)
  unsigned* claim;          // [3], zero between passes: recent-row and selected-row chunks
                            // handed out, blocks finished (the kernel clears all three when it ends)
};

int gather_cpl(int row_bytes);  // 16-byte chunks per lane of a half-warp row copy
cudaError_t launch_gather(const GatherArgs& a, cudaStream_t st);

// Appending whole frames to a streaming cache (append.cu).
struct AppendArgs {
  const void* k_new;   // [S][n_new][row_bytes], contiguous
  const void* v_new;
  void* k_dst;         // [S][cap][row_bytes]: rows row0 .. row0 + n_new - 1 written
  void* v_dst;
  uint16_t* pid;       // [S][cap] or nullptr
  uint32_t* fid;       // [S][cap] or nullptr
  int64_t n_slabs, cap, row0, n_new;
  int row_bytes, p;
  uint32_t first_frame;
  int num_sms;
};
cudaError_t launch_append(const AppendArgs& a, cudaStream_t st);

// Shared index set: per-token TaR and VaN of a layer from its heads' partial
// sums (combine.cu).
struct CombineArgs {
  const float* dot;  // [L*hs][n_tokens] per head-slab: k.m_q
  const float* kk;   //                                |k|^2
  const float* vv;   //                                |v|^2
  float* tar;        // [L][n_tokens]: rows [0, n_past) written
  float* van;
  int64_t n_layers, n_tokens, n_past;
  int hs;
  int num_sms;
};
cudaError_t launch_combine(const CombineArgs& a, cudaStream_t st);

// Layer-adaptive pooling of VaN (pool.cu): one block per slab.
constexpr int kPoolThreads = 1024;
constexpr int kMaxPoolFrame = 4096;  // IPV_MAX_POOL_FRAME_TOKENS
struct PoolArgs {
  const float* van;          // [S][n_tokens] VaN of every cached row
  float* pooled;             // [S][n_tokens]: rows [0, n_rows) written
  int32_t* pool_size;        // [S / n_heads] or nullptr
  const uint16_t* patch_id;  // [S][id_stride] or nullptr (then frame_id is nullptr too)
  const uint32_t* frame_id;
  int64_t id_stride;
  int64_t n_slabs, n_tokens, n_rows;
  int n_heads, grid_h, grid_w;
  float tau[3];
};
size_t pool_smem_bytes(int grid_h, int grid_w, bool staged);  // 0 if a frame does not fit

// Frame-level TaR ablation: each past row's score becomes its frame's mean.
struct FrameMeanArgs {
  float* tar;                // [units][n_tokens], rows [0, n_past) rewritten in place
  const uint32_t* frame_id;  // [units][id_stride] or nullptr (frame = n div p)
  int64_t id_stride;
  int64_t units, n_tokens, n_past;
  int p;
};
cudaError_t launch_frame_mean(const FrameMeanArgs& a, cudaStream_t st);
cudaError_t pool_prepare();
cudaError_t launch_pool(const PoolArgs& a, cudaStream_t st, bool pdl);

// Fused pass (window.cu): one cooperative persistent kernel, streaming
// blocks and owner blocks. Its counters live in library scratch, are zero
// before a launch and are reset by the kernel's last block.
struct WinState {      // counters first: a failed launch clears them up to `error`
  unsigned head;      // next score item (slab-major)
  unsigned sel_head;  // next slab for an owner block
  unsigned exited;    // blocks that have left
  unsigned gat_low;   // slabs below have all their gather items handed out
  unsigned error;     // bit 0: an owner gave up waiting for its slab's scores,
                      // bit 1: a streaming block gave up waiting for work
  unsigned pad[3];
};
constexpr int kWinFlags = 3;  // per-slab words: score items done, selection done, gather items handed out
constexpr size_t kWinSmemMax = 112 * 1024;  // two blocks per SM
constexpr int kWinBlock = 512;  // threads of a fused-pass block
constexpr int kWinRegE = 18;    // past tokens per owner thread: the selection's keys stay in registers

struct WinArgs {
  ScoreArgs sc;      // k, v, tar, van: the source half and library score scratch
  SelectArgs se;
  GatherArgs ga;
  WinState* state;
  unsigned* flags;   // [kWinFlags][n_slabs]
  int n_si;          // score items per slab (patch ranges)
  int qmax;          // most patches in one score item
  int n_gi, rows_gi; // gather items per slab, selected rows per gather item
  int lag;           // window: score items run at most this many slabs ahead of the
                     // oldest slab whose gather items are not all handed out
  int n_stream, n_owner;  // blocks of each kind
  int64_t spin_limit;
};

size_t window_smem_bytes(int qmax, int D, int elem, int r, int64_t n_past);
cudaError_t window_prepare();
cudaError_t window_blocks_per_sm(const WinArgs& a, size_t smem, int* per_sm);
cudaError_t launch_window(const WinArgs& a, size_t smem, cudaStream_t st);

}  // namespace ipv
