// The whole compression pass as one persistent kernel whose compaction finds
// the kept rows still in L2.
//
// The step kernels read every K and V row once to score it (Sec. 3.1 Eq. tar,
// Sec. 3.2) and then read the kept rows a second time, from HBM, to compact
// them (Sec. 3.1 K~ = K[:, I, :]; Algorithm 2 last step): about 1.4 times
// the bytes the pass has to move. Here the pass runs slab by slab over the
// whole GPU, so that a slab's rows are compacted a few slabs after they were
// scored, while they are still in the 126 MB L2.
//
// Two kinds of blocks run together, one of each per SM (a cooperative launch
// keeps them all resident, so that their waits on one another end):
//
//   streaming blocks work on two kinds of items. Score items (a slab's past
//     rows, one item per range of patches: rows f p + q of a cache that has
//     never been compacted) come from one counter in slab order; a score
//     item computes m_q of its own patches from their r recent K rows (the
//     step kernels' arithmetic), so no block waits for another's means.
//     Gather items (a slab's selected past rows, copied to the other
//     ping-pong half) come from a per-slab counter once the slab's
//     selection is done. Warp 0 of a block picks the block's next item: a
//     ready gather item first (the lowest such slab), else the score item it
//     holds. A block claims its next score item ahead, and copies that
//     item's recent rows into shared memory while the current item runs,
//     only while it lies within `window` slabs of the oldest slab whose
//     gather items are not all handed out: so the rows of at most about
//     `window` slabs wait in L2 for their compaction. A block never waits
//     while it holds a score item.
//   owner blocks take slabs in order. For its slab an owner copies the
//     recent rows (always kept) to their final place, waits until the slab's
//     score items are done, and runs the split-budget selection (Sec. 3.3;
//     Algorithm 1 steps 3-5) into kept_idx.
//
// Data produced inside the kernel (scores, kept indices) is published by
// __syncthreads, a fence and a counter update, and read after an acquire
// load through L2. K and V sources are never written (the destination is the
// other half) and use non-coherent loads. Every wait is bounded: on timeout
// the block sets a bit in the state's error word and goes on with whatever
// the awaited data holds (the results are then invalid; no access leaves its
// buffer). The last block out resets the counters for the next pass.
#include "pass_device.cuh"

namespace ipv {
namespace {

constexpr int kWinThreads = 512;
static_assert(kWinThreads == ipv::kWinBlock, "fused block size");

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Thread 0: bounded wait until *p >= want; false if it gave up.
__device__ bool wait_at_least(const unsigned* p, unsigned want, int64_t limit) {
  for (int64_t spins = 0; ld_acquire(p) < want; ++spins) {
    if (spins >= limit) return false;
    __nanosleep(128);
  }
  return true;
}

// Thread 0, after the block's __syncthreads: make the block's writes visible
// before the counter moves.
__device__ __forceinline__ void release_add(unsigned* p, unsigned v) {
  __threadfence();
  atomicAdd(p, v);
}

__device__ __forceinline__ unsigned ld_relaxed(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

struct Item {  // a score item
  int kind;    // 1
  int s, k;    // slab, item within the slab
};

// What a streaming block does next (decided by warp 0).
enum { kIdle = 0, kGather = 1, kScoreHeld = 2, kScoreNew = 3, kExit = 4 };

// Score item k of a slab covers patches [k p / n_si, (k + 1) p / n_si).
__device__ __forceinline__ int item_q0(const WinArgs& a, int k) { return k * a.sc.p / a.n_si; }

// Issues 16-byte asynchronous copies of the recent K rows of a score item's
// patches into krec (row t' nq + (q - q0) holds row n_past + t' p + q) and
// commits them as one group; every thread of the block takes a share.
__device__ __forceinline__ void prefetch_recent(const WinArgs& a, const Item& it, char* krec, int row_bytes) {
  const int q0 = item_q0(a, it.k), nq = item_q0(a, it.k + 1) - q0;
  const int n_chunks = row_bytes / 16;
  const int64_t n_past = a.sc.n_tokens - static_cast<int64_t>(a.sc.r) * a.sc.p;
  const char* kslab = static_cast<const char*>(a.sc.k) + static_cast<int64_t>(it.s) * a.sc.cap * row_bytes;
  const int total = a.sc.r * nq * n_chunks;
  for (int i = threadIdx.x; i < total; i += blockDim.x) {
    const int row = i / n_chunks, c = i - row * n_chunks;
    const int t = row / nq, q = q0 + (row - t * nq);
    cp_async16(krec + static_cast<int64_t>(row) * row_bytes + c * 16,
               kslab + (n_past + static_cast<int64_t>(t) * a.sc.p + q) * row_bytes + c * 16);
  }
  asm volatile("cp.async.commit_group;" ::: "memory");
}

// m_q of a score item's nq patches from their recent K rows in krec (Sec. 3.1
// Eq. tar, regrouped: m_q = (1/r) sum_t' k_t' / max(|k_t'|, eps)), into mtab
// rows of ms floats. The arithmetic of dev::mean_group: per row a lane group
// sums |k|^2 over its chunks in order, then each patch's group accumulates
// the normalised rows t' = 0, 1, ... with one fma per element. Ends with a
// __syncthreads.
template <typename T, int LPR, int CPL>
__device__ __forceinline__ void item_mean(const WinArgs& a, int nq, const char* krec, float* rinv,
                                          float* mtab, int ms) {
  constexpr int P2 = Chunk<T>::kPairs;
  constexpr int E = Chunk<T>::kElems;
  constexpr int RPW = 32 / LPR;
  const int lane = threadIdx.x & 31, sub = lane % LPR;
  const int g = (threadIdx.x >> 5) * RPW + lane / LPR, G = (blockDim.x >> 5) * RPW;
  const int row_bytes = a.sc.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int rows = a.sc.r * nq;
  for (int base = 0; base < rows; base += G) {  // warp-uniform: 1 / max(|k|, eps) of each row
    const int row = base + g;
    float2 kk2 = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
      const int c = sub + LPR * i;
      const uint4 raw = (row < rows && c < n_chunks)
                            ? *reinterpret_cast<const uint4*>(krec + static_cast<int64_t>(row) * row_bytes + c * 16)
                            : make_uint4(0, 0, 0, 0);
      float2 x[P2];
      Chunk<T>::widen2(raw, x);
#pragma unroll
      for (int e = 0; e < P2; ++e) kk2 = fma2(x[e], x[e], kk2);
    }
    const float kk = dev::group_sum<LPR>(kk2.x + kk2.y);
    if (row < rows && sub == 0) rinv[row] = rsqrtf(fmaxf(kk, kNormEps * kNormEps));
  }
  __syncthreads();
  if (g < nq) {
    float2 acc[CPL][P2];
#pragma unroll
    for (int i = 0; i < CPL; ++i)
#pragma unroll
      for (int e = 0; e < P2; ++e) acc[i][e] = make_float2(0.0f, 0.0f);
    for (int t = 0; t < a.sc.r; ++t) {
      const int row = t * nq + g;
      const float inv = rinv[row];
      const float2 inv2 = make_float2(inv, inv);
#pragma unroll
      for (int i = 0; i < CPL; ++i) {
        const int c = sub + LPR * i;
        const uint4 raw = c < n_chunks
                              ? *reinterpret_cast<const uint4*>(krec + static_cast<int64_t>(row) * row_bytes + c * 16)
                              : make_uint4(0, 0, 0, 0);
        float2 x[P2];
        Chunk<T>::widen2(raw, x);
#pragma unroll
        for (int e = 0; e < P2; ++e) acc[i][e] = fma2(x[e], inv2, acc[i][e]);
      }
    }
    const float inv_r = 1.0f / static_cast<float>(a.sc.r);
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
      const int c = sub + LPR * i;
      if (c < n_chunks) {
        float* mrow = mtab + g * ms + c * E;
#pragma unroll
        for (int e = 0; e < P2; e += 2)
          *reinterpret_cast<float4*>(mrow + 2 * e) =
              make_float4(acc[i][e].x * inv_r, acc[i][e].y * inv_r, acc[i][e + 1].x * inv_r,
                          acc[i][e + 1].y * inv_r);
      }
    }
  }
  __syncthreads();
}

template <typename T, int LPR, int CPL, int GCPL>
__global__ void __launch_bounds__(kWinThreads, 2) window_kernel(WinArgs a) {
  extern __shared__ __align__(16) uint32_t sm[];
  __shared__ dev::SelShared sh;
  __shared__ unsigned s_tk[1];
  __shared__ unsigned s_cmd[3];
  __shared__ int s_last;
  constexpr int kGU = GCPL >= 4 ? 1 : 4 / GCPL;  // rows in flight per half-warp
  WinState* st = a.state;
  const int S = static_cast<int>(a.sc.n_slabs);
  unsigned* s_count = a.flags;      // score items finished
  unsigned* x_done = a.flags + S;   // selection finished
  unsigned* g_next = a.flags + 2 * S;  // gather items handed out
  const int64_t rp = static_cast<int64_t>(a.sc.r) * a.sc.p;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;

  if (blockIdx.x < a.n_stream) {
    // ------------------------------------------------------------ streaming
    const unsigned total_s = static_cast<unsigned>(S) * a.n_si;  // score tickets
    const int f_past = static_cast<int>((a.sc.n_tokens - rp) / a.sc.p);
    const int row_bytes = a.sc.D * static_cast<int>(sizeof(T));
    const int ms = a.sc.D + 4;  // padded m rows: lane groups of different patches hit different banks
    const int rec_rows = a.sc.r * a.qmax;
    char* krec[2] = {reinterpret_cast<char*>(sm),
                     reinterpret_cast<char*>(sm) + static_cast<int64_t>(rec_rows) * row_bytes};
    float* mtab = reinterpret_cast<float*>(krec[1] + static_cast<int64_t>(rec_rows) * row_bytes);
    float* rinv = mtab + a.qmax * ms;
    const unsigned kNone = 0xFFFFFFFFu;
    unsigned held = kNone;  // score ticket claimed ahead, its recent rows in krec[hbuf]
    int hbuf = 0;
    int64_t idle = 0;
    for (;;) {
      if (warp == 0) {
        int kind = kIdle;
        unsigned id = 0u, nxt = kNone;
        // A ready gather item: lane l looks at slab gat_low + l.
        const unsigned gl = ld_relaxed(&st->gat_low);
        const unsigned sl = gl + lane;
        const bool in = sl < static_cast<unsigned>(S);
        const unsigned gn = in ? ld_relaxed(&g_next[sl]) : 0xFFFFFFFFu;
        const bool ready = in && gn < static_cast<unsigned>(a.n_gi) && ld_acquire(&x_done[sl]) != 0u;
        unsigned mask = __ballot_sync(0xffffffffu, ready);
        while (mask) {
          const int l = __ffs(mask) - 1;
          unsigned c = 0u;
          if (lane == l) c = atomicAdd(&g_next[sl], 1u);
          c = __shfl_sync(0xffffffffu, c, l);
          if (c < static_cast<unsigned>(a.n_gi)) {
            kind = kGather;
            id = (gl + l) * static_cast<unsigned>(a.n_gi) + c;
            break;
          }
          mask &= mask - 1u;
        }
        // Move the watermark over slabs whose gather items are all handed out.
        const unsigned open = __ballot_sync(0xffffffffu, !(in && gn >= static_cast<unsigned>(a.n_gi)));
        const unsigned skip = open ? static_cast<unsigned>(__ffs(open) - 1) : 32u;
        if (lane == 0) {
          if (skip > 0u) atomicMax(&st->gat_low, gl + skip);
          // Else the held score item, or a new one within the window; and
          // the next one ahead, within the window.
          auto claim = [&]() -> unsigned {
            const unsigned h = ld_relaxed(&st->head);
            if (h >= total_s || h / a.n_si >= gl + skip + a.lag) return kNone;
            const unsigned t = atomicAdd(&st->head, 1u);
            return t < total_s ? t : kNone;
          };
          if (kind == kIdle) {
            if (held != kNone) {
              kind = kScoreHeld;
              id = held;
            } else if ((id = claim()) != kNone) {
              kind = kScoreNew;
            }
            if (kind != kIdle) nxt = claim();
          }
          if (kind == kIdle && held == kNone && ld_relaxed(&st->head) >= total_s &&
              gl + skip >= static_cast<unsigned>(S))
            kind = kExit;
          s_cmd[0] = static_cast<unsigned>(kind);
          s_cmd[1] = id;
          s_cmd[2] = nxt;
        }
      }
      __syncthreads();
      const int kind = static_cast<int>(s_cmd[0]);
      const unsigned id = s_cmd[1], nxt = s_cmd[2];
      if (kind == kExit) break;
      if (kind == kIdle) {
        if (++idle > a.spin_limit) {  // nothing became ready: give up rather than hang
          if (threadIdx.x == 0) atomicOr(&st->error, 2u);
          break;
        }
        __nanosleep(256);
        __syncthreads();  // s_cmd is rewritten next round
        continue;
      }
      idle = 0;
      if (kind == kGather) {
        const int s = static_cast<int>(id / a.n_gi), c = static_cast<int>(id % a.n_gi);
        const int64_t j0 = static_cast<int64_t>(c) * a.rows_gi;
        const int64_t j1 = min(a.se.budget - rp, j0 + a.rows_gi);
        const int64_t base = static_cast<int64_t>(s) * a.se.budget;
        dev::gather_range<GCPL, kGU, true, false, true>(a.ga, base + j0, base + j1, threadIdx.x >> 4,
                                                        blockDim.x >> 4);
        __syncthreads();
        continue;
      }
      // A score item: its recent rows (copied now if they were not claimed
      // ahead), and the next item's rows into the other buffer meanwhile.
      const Item it{1, static_cast<int>(id / a.n_si), static_cast<int>(id % a.n_si)};
      if (kind == kScoreNew) prefetch_recent(a, it, krec[hbuf], row_bytes);
      if (nxt != kNone) {
        const Item nt{1, static_cast<int>(nxt / a.n_si), static_cast<int>(nxt % a.n_si)};
        prefetch_recent(a, nt, krec[hbuf ^ 1], row_bytes);
        asm volatile("cp.async.wait_group 1;" ::: "memory");  // this item's rows, not the next's
      } else {
        cp_async_wait_all();
      }
      __syncthreads();
      const int q0 = item_q0(a, it.k), nq = item_q0(a, it.k + 1) - q0;
      item_mean<T, LPR, CPL>(a, nq, krec[hbuf], rinv, mtab, ms);
      dev::score_patch_rows<T, LPR, CPL>(a.sc, it.s, q0, nq, f_past, mtab, ms);
      __syncthreads();
      if (threadIdx.x == 0) release_add(&s_count[it.s], 1u);
      held = nxt;
      if (nxt != kNone) hbuf ^= 1;
    }
    cp_async_wait_all();
  } else {
    // ------------------------------------------------------------ owners
    for (;;) {
      if (threadIdx.x == 0) s_tk[0] = atomicAdd(&st->sel_head, 1u);
      __syncthreads();
      const unsigned s = s_tk[0];
      __syncthreads();
      if (s >= static_cast<unsigned>(S)) break;
      // The recent rows are always kept: copy them to rows budget - rp + j.
      dev::gather_range<GCPL, kGU, true, true, true>(a.ga, static_cast<int64_t>(s) * rp,
                                                     static_cast<int64_t>(s + 1) * rp, threadIdx.x >> 4,
                                                     blockDim.x >> 4, rp);
      if (threadIdx.x == 0 && !wait_at_least(&s_count[s], static_cast<unsigned>(a.n_si), a.spin_limit))
        atomicOr(&st->error, 1u);
      __syncthreads();
      dev::select_slab_reg<kWinThreads, kWinRegE>(a.se, s, sm, sh);
      if (threadIdx.x == 0) release_add(&x_done[s], 1u);
    }
  }

  // Leave; the last block out resets the counters for the next pass.
  __syncthreads();
  if (threadIdx.x == 0) {
    __threadfence();
    s_last = (atomicAdd(&st->exited, 1u) == gridDim.x - 1u) ? 1 : 0;
  }
  __syncthreads();
  if (s_last) {
    __threadfence();
    for (int i = threadIdx.x; i < kWinFlags * S; i += blockDim.x) a.flags[i] = 0u;
    if (threadIdx.x == 0) {
      st->head = 0u;
      st->sel_head = 0u;
      st->gat_low = 0u;
      st->exited = 0u;
    }
    __threadfence();
  }
}

template <typename T, int LPR, int CPL, int GCPL>
cudaError_t run(const WinArgs& a, size_t smem, int grid, cudaStream_t stream, bool prepare,
                int* per_sm) {
  auto kern = window_kernel<T, LPR, CPL, GCPL>;
  if (prepare)
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(kWinSmemMax));
  if (per_sm) return cudaOccupancyMaxActiveBlocksPerMultiprocessor(per_sm, kern, kWinThreads, smem);
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(grid);
  cfg.blockDim = dim3(kWinThreads);
  cfg.dynamicSmemBytes = smem;
  cfg.stream = stream;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeCooperative;  // every block resident at once
  attr[0].val.cooperative = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, a);
}

template <typename T>
cudaError_t dispatch(const WinArgs& a, size_t smem, int grid, cudaStream_t st, bool prepare, int shape,
                     int* per_sm) {
  // Row shapes by 16-byte chunks per row (lanes per row, chunks per lane) of
  // the scoring, as in the step kernels, and chunks per half-warp lane of
  // the compaction.
  switch (shape) {
    case 41: return run<T, 4, 1, 1>(a, smem, grid, st, prepare, per_sm);
    case 42: return run<T, 4, 2, 1>(a, smem, grid, st, prepare, per_sm);
    case 44: return run<T, 4, 4, 1>(a, smem, grid, st, prepare, per_sm);
    case 84: return run<T, 8, 4, 2>(a, smem, grid, st, prepare, per_sm);
    case 164: return run<T, 16, 4, 4>(a, smem, grid, st, prepare, per_sm);
    default: return run<T, 16, 8, 8>(a, smem, grid, st, prepare, per_sm);
  }
}

}  // namespace

size_t window_smem_bytes(int qmax, int D, int elem, int r, int64_t n_past) {
  const size_t rec = static_cast<size_t>(r) * qmax;  // recent rows of one score item
  const size_t stream_b = 2 * rec * D * elem + static_cast<size_t>(qmax) * (D + 4) * sizeof(float) +
                          rec * sizeof(float);
  const size_t owner_b = dev::select_reg_smem_words<kWinThreads, kWinRegE>() * sizeof(uint32_t);
  return stream_b > owner_b ? stream_b : owner_b;
}

cudaError_t window_prepare() {
  const int shapes[] = {41, 42, 44, 84, 164, 168};
  for (int shape : shapes) {
    WinArgs a{};
    cudaError_t e = dispatch<uint16_t>(a, 0, 0, nullptr, true, shape, nullptr);
    if (e != cudaSuccess) return e;
    e = dispatch<float>(a, 0, 0, nullptr, true, shape, nullptr);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t window_blocks_per_sm(const WinArgs& a, size_t smem, int* per_sm) {
  const int shape = row_shape(a.sc.D, a.sc.is_bf16);
  return a.sc.is_bf16 ? dispatch<uint16_t>(a, smem, 0, nullptr, false, shape, per_sm)
                      : dispatch<float>(a, smem, 0, nullptr, false, shape, per_sm);
}

cudaError_t launch_window(const WinArgs& a, size_t smem, cudaStream_t st) {
  const int shape = row_shape(a.sc.D, a.sc.is_bf16);
  const int grid = a.n_stream + a.n_owner;
  return a.sc.is_bf16 ? dispatch<uint16_t>(a, smem, grid, st, false, shape, nullptr)
                      : dispatch<float>(a, smem, grid, st, false, shape, nullptr);
}

}  // namespace ipv
