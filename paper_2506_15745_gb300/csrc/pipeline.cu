// The whole compression pass as one persistent kernel.
//
// The four steps of the pass (recent-frame mean, TaR/VaN scoring, split-
// budget selection, compaction; InfiniPot-V Sec. 3.1-3.3, Algorithms 1-2) are
// cut into work items that one block per SM takes from device-side queues:
//
//   main queue    : recent-mean items (one per slab) and score items (one per
//                   chunk of a slab's past rows), grouped so that the means of a
//                   group are queued `lead` groups before its score chunks;
//   selections    : one item per slab, taken once all its score chunks are done;
//   gathers       : chunks of a slab's kept rows, taken once its selection is done.
//
// Selections and gathers are handed out per slab: warp 0 of a block looks at
// the 32 slabs above a watermark at once and claims a ready one with a single
// atomic (an exchange for a selection, a ticket for a gather chunk), so
// claims never retry and idle blocks do not serialise on a shared head.
//
// A block prefers ready gather items, then ready select items, then the main
// queue. Selections (latency-bound shared-memory work) thus overlap the HBM
// streams of other blocks, and a slab's rows are copied soon after they were
// scored, while many of them are still in L2. Only a score item can wait
// (for its slab's mean, which an earlier, running block has taken); select and
// gather items are taken only when ready. Every wait is bounded: on timeout
// the block records it in the state's error word and carries on or leaves.
//
// Data produced inside the kernel (m, scores, kept indices) is published by
// __syncthreads, a fence and a release counter update, and read after an
// acquire load with ordinary loads. The K/V sources are never written by the
// kernel (the destination is the other ping-pong half) and use .nc loads.
#include "pass_device.cuh"

namespace ipv {
namespace {

constexpr int kPipeThreads = 512;

enum ItemKind { kNone = 0, kGather = 1, kSelect = 2, kMain = 3, kWait = 4, kExit = 5 };

__device__ __forceinline__ unsigned ld_acquire(const unsigned* p) {
  unsigned v;
  asm volatile("ld.acquire.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

__device__ __forceinline__ unsigned ld_relaxed(const unsigned* p) {
  unsigned v;
  asm volatile("ld.relaxed.gpu.global.u32 %0, [%1];" : "=r"(v) : "l"(p) : "memory");
  return v;
}

// Called by thread 0 after the block's __syncthreads: publish the item's writes.
__device__ __forceinline__ void release_add(unsigned* p, unsigned v) {
  __threadfence();
  atomicAdd(p, v);
}

template <typename T, int LPR, int CPL, int GCPL, int BLPR, int BCPL>
__global__ void __launch_bounds__(kPipeThreads, 1) pipeline_kernel(PipeArgs a) {
  extern __shared__ __align__(128) uint32_t sm_sel[];
  __shared__ dev::SelShared sh;
  __shared__ dev::BulkRing ring;
  __shared__ int s_kind;
  __shared__ int s_id;
  constexpr int RPW = 32 / LPR;
  constexpr int kScoreU = CPL >= 8 ? 1 : 2;
  constexpr int kGatherU = GCPL >= 4 ? 2 : 8 / GCPL;
  PipeState* st = a.state;
  const int S = static_cast<int>(a.sc.n_slabs);
  unsigned* m_done = a.flags;            // recent mean written
  unsigned* s_count = a.flags + S;       // score chunks finished
  unsigned* x_claim = a.flags + 2 * S;   // selection taken by a block
  unsigned* x_done = a.flags + 3 * S;    // selection finished
  unsigned* g_next = a.flags + 4 * S;    // gather chunks handed out
  const int n_past = static_cast<int>(a.sc.n_tokens - static_cast<int64_t>(a.sc.r) * a.sc.p);
  const int block_items = a.group * (1 + a.n_sc);
  const unsigned n_main = static_cast<unsigned>((a.n_groups + a.lead) * block_items);
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  int64_t idle = 0;
  // Score chunks: the slab's m table and a ring of bulk-copy stages share the
  // dynamic shared memory with the selection (one item at a time).
  float* m_tab = reinterpret_cast<float*>(sm_sel);
  const int m_floats = a.sc.p * a.sc.D;
  char* stages = reinterpret_cast<char*>(m_tab + ((m_floats + 31) & ~31));
  uint32_t seq = 0;
  if (threadIdx.x == 0 && a.nst >= 2) dev::ring_init(ring, a.nst);
  __syncthreads();

  for (;;) {
    if (warp == 0) {
      // Warp 0 picks the block's next item. Lane l looks at slab low + l of
      // the gather and select windows; a claim is one atomic that cannot fail
      // (a ticket), so many idle blocks never serialise on a compare-and-swap.
      int kind = kNone, id = 0;
      const unsigned gl = ld_relaxed(&st->gat_low);
      {
        const unsigned s = gl + lane;
        const bool in = s < static_cast<unsigned>(S);
        const unsigned gn = in ? ld_relaxed(&g_next[s]) : 0xFFFFFFFFu;
        const bool ready = in && gn < static_cast<unsigned>(a.n_ga) && ld_relaxed(&x_done[s]) != 0u;
        unsigned mask = __ballot_sync(0xffffffffu, ready);
        while (mask) {
          const int l = __ffs(mask) - 1;
          unsigned c = 0u;
          if (lane == l) c = atomicAdd(&g_next[s], 1u);
          c = __shfl_sync(0xffffffffu, c, l);
          if (c < static_cast<unsigned>(a.n_ga)) {
            kind = kGather;
            id = static_cast<int>((gl + l) * a.n_ga + c);
            break;
          }
          mask &= mask - 1u;
        }
        // Advance the watermark over slabs whose chunks are all handed out.
        const unsigned open = __ballot_sync(0xffffffffu, !(in && gn >= static_cast<unsigned>(a.n_ga)));
        const unsigned skip = open ? static_cast<unsigned>(__ffs(open) - 1) : 32u;
        if (lane == 0 && skip > 0u) atomicMax(&st->gat_low, gl + skip);
      }
      if (kind == kNone) {
        const unsigned xl = ld_relaxed(&st->sel_low);
        const unsigned s = xl + lane;
        const bool in = s < static_cast<unsigned>(S);
        const unsigned claimed = in ? ld_relaxed(&x_claim[s]) : 1u;
        const bool ready = in && claimed == 0u && ld_relaxed(&s_count[s]) == static_cast<unsigned>(a.n_sc);
        unsigned mask = __ballot_sync(0xffffffffu, ready);
        while (mask) {
          const int l = __ffs(mask) - 1;
          unsigned old = 1u;
          if (lane == l) old = atomicExch(&x_claim[s], 1u);
          old = __shfl_sync(0xffffffffu, old, l);
          if (old == 0u) {
            kind = kSelect;
            id = static_cast<int>(xl + l);
            break;
          }
          mask &= mask - 1u;
        }
        const unsigned open = __ballot_sync(0xffffffffu, !(in && claimed != 0u));
        const unsigned skip = open ? static_cast<unsigned>(__ffs(open) - 1) : 32u;
        if (lane == 0 && skip > 0u) atomicMax(&st->sel_low, xl + skip);
      }
      if (lane == 0) {
        if (kind == kNone && ld_relaxed(&st->main_head) < n_main) {
          const unsigned hm = atomicAdd(&st->main_head, 1u);
          if (hm < n_main) {
            kind = kMain;
            id = static_cast<int>(hm);
          }
        }
        if (kind == kNone) kind = ld_relaxed(&st->gat_low) >= static_cast<unsigned>(S) ? kExit : kWait;
        // The flags behind a gather or select claim were read relaxed: this
        // fence makes the producer's writes visible before the block reads them.
        if (kind == kGather || kind == kSelect) __threadfence();
        s_kind = kind;
        s_id = id;
      }
    }
    __syncthreads();
    const int kind = s_kind, id = s_id;
    __syncthreads();
    if (kind == kExit) break;
    if (kind == kWait) {
      if (++idle > a.spin_limit) {  // nothing became ready: give up rather than hang
        if (threadIdx.x == 0) atomicOr(&st->error, 2u);
        break;
      }
      __nanosleep(256);
      continue;
    }
    idle = 0;

    if (kind == kGather) {
      const int s = id / a.n_ga, c = id - s * a.n_ga;
      const int64_t j0 = static_cast<int64_t>(c) * a.rows_ga;
      const int64_t j1 = min(static_cast<int64_t>(a.se.budget), j0 + a.rows_ga);
      const int64_t base = static_cast<int64_t>(s) * a.se.budget;
      dev::gather_range<GCPL, kGatherU>(a.ga, base + j0, base + j1, threadIdx.x >> 4,
                                        blockDim.x >> 4);
      continue;  // nothing waits on gathers
    }

    if (kind == kSelect) {
      dev::select_slab<kPipeThreads>(a.se, id, sm_sel, sh);
      __syncthreads();
      if (threadIdx.x == 0) release_add(&x_done[id], 1u);
      continue;
    }

    // Main queue item: decode (block of `group` means, then score chunks of
    // the group `lead` blocks earlier).
    const int blk = id / block_items, r = id - blk * block_items;
    if (r < a.group) {
      const int s = blk * a.group + r;
      if (blk >= a.n_groups || s >= S) continue;  // padding slot
      for (int q0 = warp * RPW; q0 < a.sc.p; q0 += n_warps * RPW) {  // warp-uniform
        const int q = q0 + lane / LPR;
        dev::mean_group<T, LPR, CPL>(a.sc, s, q < a.sc.p ? q : 0, q < a.sc.p);
      }
      __syncthreads();
      if (threadIdx.x == 0) release_add(&m_done[s], 1u);
      continue;
    }
    const int g = blk - a.lead;
    const int idx = r - a.group;
    const int s = g * a.group + idx / a.n_sc, c = idx % a.n_sc;
    if (g < 0 || s >= S) continue;  // padding slot
    if (threadIdx.x == 0) {
      int64_t spins = 0;
      while (ld_acquire(&m_done[s]) == 0u) {
        if (++spins > a.spin_limit) {
          atomicOr(&st->error, 1u);
          break;
        }
        __nanosleep(128);
      }
    }
    __syncthreads();
    const int lo = c * a.rows_sc;
    const int hi = min(n_past, lo + a.rows_sc);
    const float* m_slab = a.sc.m + static_cast<int64_t>(s) * m_floats;
    if (a.nst >= 2) {
      dev::load_m_planes<T, false>(m_slab, m_tab, a.sc.p, a.sc.D);  // written in this kernel
      __syncthreads();
      dev::score_segment_bulk<T, BLPR, BCPL>(a.sc, s, lo, hi, m_tab, stages, a.nst, ring, seq);
    } else {
      dev::score_segment<T, LPR, CPL, kScoreU, dev::kMGlobal>(a.sc, s, lo, hi, m_slab, a.sc.D);
    }
    __syncthreads();
    if (threadIdx.x == 0) release_add(&s_count[s], 1u);
  }

  // Leave; the last block out resets the queue state for the next pass.
  __syncthreads();
  if (threadIdx.x == 0) s_kind = (atomicAdd(&st->exited, 1u) == gridDim.x - 1u) ? 1 : 0;
  __syncthreads();
  if (s_kind) {
    __threadfence();
    for (int i = threadIdx.x; i < kPipeFlags * S; i += blockDim.x) a.flags[i] = 0u;
    if (threadIdx.x == 0) {
      st->main_head = 0u;
      st->sel_low = 0u;
      st->gat_low = 0u;
      st->exited = 0u;
    }
  }
}

template <typename T, int LPR, int CPL, int GCPL, int BLPR, int BCPL>
cudaError_t run(const PipeArgs& a, size_t smem, int num_sms, cudaStream_t stream, bool prepare) {
  auto kern = pipeline_kernel<T, LPR, CPL, GCPL, BLPR, BCPL>;
  if (prepare)
    return cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                static_cast<int>(kBulkSmemMax));
  kern<<<num_sms, kPipeThreads, smem, stream>>>(a);
  return cudaGetLastError();
}

template <typename T>
cudaError_t dispatch(const PipeArgs& a, size_t smem, int num_sms, cudaStream_t st, bool prepare,
                     int shape) {
  // Row shapes by 16-byte chunks per row: (lanes per row, chunks per lane) of
  // the load-based scoring and of the bulk-copy scoring, and chunks per
  // half-warp lane of the compaction.
  switch (shape) {
    case 41: return run<T, 4, 1, 1, 8, 1>(a, smem, num_sms, st, prepare);
    case 42: return run<T, 4, 2, 1, 8, 1>(a, smem, num_sms, st, prepare);
    case 44: return run<T, 4, 4, 1, 8, 2>(a, smem, num_sms, st, prepare);
    case 84: return run<T, 8, 4, 2, 8, 4>(a, smem, num_sms, st, prepare);
    case 164: return run<T, 16, 4, 4, 16, 4>(a, smem, num_sms, st, prepare);
    default: return run<T, 16, 8, 8, 32, 4>(a, smem, num_sms, st, prepare);
  }
}

}  // namespace

size_t pipeline_smem_bytes(int64_t n_past) {
  return dev::select_smem_words<kPipeThreads>(n_past) * sizeof(uint32_t);
}

int pipeline_stages(int p, int D, int elem) { return bulk_stages(p, D, elem, kPipeThreads); }

cudaError_t pipeline_prepare() {
  const int shapes[] = {41, 42, 44, 84, 164, 168};
  for (int shape : shapes) {
    PipeArgs a{};
    cudaError_t e = dispatch<uint16_t>(a, 0, 0, nullptr, true, shape);
    if (e != cudaSuccess) return e;
    e = dispatch<float>(a, 0, 0, nullptr, true, shape);
    if (e != cudaSuccess) return e;
  }
  return cudaSuccess;
}

cudaError_t launch_pipeline(const PipeArgs& a, int num_sms, cudaStream_t st) {
  const int64_t n_past = a.sc.n_tokens - static_cast<int64_t>(a.sc.r) * a.sc.p;
  const int elem = a.sc.is_bf16 ? 2 : 4;
  size_t smem = pipeline_smem_bytes(n_past);
  if (a.nst >= 2) {
    const size_t b = bulk_smem_bytes(a.sc.p, a.sc.D, elem, a.nst, kPipeThreads);
    smem = b > smem ? b : smem;
  }
  const int shape = row_shape(a.sc.D, a.sc.is_bf16);
  return a.sc.is_bf16 ? dispatch<uint16_t>(a, smem, num_sms, st, false, shape)
                      : dispatch<float>(a, smem, num_sms, st, false, shape);
}

}  // namespace ipv
