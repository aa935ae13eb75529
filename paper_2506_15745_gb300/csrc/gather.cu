// Step (iv) of the compression pass: compaction of the kept rows.
//
// InfiniPot-V Sec. 3.1 / Algorithm 2 last step: K~ = K[:, J, :], V~ = V[:, J, :]
// with J ascending, i.e. dst row j of a slab is src row kept[j], bytes
// unchanged. The destination is the other half of the ping-pong cache, so the
// copy has no read/write hazards and the source stays intact.
//
// Pure data movement (HBM-bound): a half-warp moves one 16-byte-chunked K row
// and the matching V row, several rows in flight per half-warp. The recent
// frames (always kept, always the last rp kept rows) are copied before the
// kernel waits for the selection, overlapping it: they are handed out in
// chunks by a device counter, so the blocks that are already resident while
// the selection runs (one beside each 1024-thread selection block, several on
// the SMs it leaves free) copy all of them. The selected rows are handed out
// the same way after the wait; one warp per block stages the next chunk's
// kept indices in shared memory (cp.async) while the block copies the
// current chunk, so no row load waits behind an index load. Patch and frame
// ids travel with their rows, copied by a separate coalesced loop.
#include "pass_device.cuh"

namespace ipv {
namespace {

constexpr int kGatherThreads = 256;   // 64 registers: one block fits beside a selection block
// Rows per claim: with rows of up to 256 bytes, one round of row loads of
// the whole block (16 half-warps x 4 rows in flight); larger chunks measured
// slower (LLaVA-OV-7B shape: 0.2015 ms at 64, 0.2043 at 128, 0.2076 at 256).
constexpr int64_t kRowChunk = 64;

// Copies the chunks of [0, total) recent rows (kRowChunk each) that the
// block claims from *counter, the next claim in flight while a chunk is
// copied. A recent row's source follows from its position, so no index is
// read.
template <int CPL, int kU>
__device__ __forceinline__ void claim_recent(const GatherArgs& a, unsigned* counter, int64_t total, int64_t jn,
                                             unsigned* s_next) {
  const int64_t n_chunks = (total + kRowChunk - 1) / kRowChunk;
  __syncthreads();  // every thread has read *s_next of an earlier call
  if (threadIdx.x == 0) *s_next = atomicAdd(counter, 1u);
  __syncthreads();
  unsigned c = *s_next;
  while (c < n_chunks) {  // block-uniform
    unsigned nxt = 0;
    if (threadIdx.x == 0) nxt = atomicAdd(counter, 1u);  // claimed ahead of need
    const int64_t b0 = static_cast<int64_t>(c) * kRowChunk;
    dev::gather_range<CPL, kU, false, true>(a, b0, min(total, b0 + kRowChunk), threadIdx.x >> 4,
                                                    blockDim.x >> 4, jn);
    __syncthreads();  // every thread has read *s_next
    if (threadIdx.x == 0) *s_next = nxt;
    __syncthreads();
    c = *s_next;
  }
}

// A claimed chunk of selected rows, staged in shared memory for the whole
// block: each row's slab s and source row n (kept[s][j], -1 past the end);
// its position j among the slab's kept rows follows from the chunk's first
// flattened row g0 as g0 + t - s jn.
struct ChunkStage {
  int32_t n[kRowChunk];
  int32_t s[kRowChunk];
};

// Warp 0 stages chunk c: the kept indices arrive by cp.async, so that no
// register waits for them while the warp copies its share of the previous
// chunk (the caller waits for them before the barrier that publishes them).
__device__ __forceinline__ void stage_chunk(const GatherArgs& a, unsigned c, int64_t total, int64_t jn,
                                            ChunkStage& st) {
  const int lane = threadIdx.x & 31;
  const int64_t g0 = static_cast<int64_t>(c) * kRowChunk + lane;
  int64_t s = g0 / jn, j = g0 - s * jn;
  for (int t = lane; t < kRowChunk; t += 32) {
    if (g0 + (t - lane) < total) {
      st.s[t] = static_cast<int32_t>(s);
      cp_async4(&st.n[t], a.kept + (a.heads_per_kept > 1 ? s / a.heads_per_kept : s) * a.budget + j);
    } else {
      st.n[t] = -1;
    }
    j += 32;  // the row 32 further on
    while (j >= jn) {
      j -= jn;
      ++s;
    }
  }
}

// Copies a staged chunk: half-warp hw takes rows hw, hw + 16, ..., kU of
// them in flight.
template <int CPL, int kU>
__device__ __forceinline__ void copy_staged(const GatherArgs& a, const ChunkStage& st, int64_t g0, int64_t jn) {
  const int hw = threadIdx.x >> 4, n_hw = blockDim.x >> 4;
  const int lane = threadIdx.x & 15;
  const int n_chunks = a.row_bytes / 16;
  const char* ks = static_cast<const char*>(a.k_src);
  const char* vs = static_cast<const char*>(a.v_src);
  char* kd = static_cast<char*>(a.k_dst);
  char* vd = static_cast<char*>(a.v_dst);
  for (int r0 = hw; r0 < kRowChunk; r0 += n_hw * kU) {
    uint4 kr[kU][CPL], vr[kU][CPL];
    int64_t dst_off[kU];
    bool ok[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int r = r0 + u * n_hw;
      const int n = r < kRowChunk ? st.n[r] : -1;
      ok[u] = n >= 0 && n < a.cap;
      const int64_t sl = ok[u] ? st.s[r] : 0;
      const int64_t base = sl * a.cap;
      dst_off[u] = (base + (ok[u] ? g0 + r - sl * jn : 0)) * a.row_bytes;
      const int64_t src_off = (base + (ok[u] ? n : 0)) * a.row_bytes;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        const bool ld = ok[u] && ch < n_chunks;
        kr[u][c] = ld ? ld_stream(ks + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
        vr[u][c] = ld ? ld_stream(vs + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      if (!ok[u]) continue;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        if (ch < n_chunks) {
          st_stream(kd + dst_off[u] + ch * 16, kr[u][c]);
          st_stream(vd + dst_off[u] + ch * 16, vr[u][c]);
        }
      }
    }
  }
}

// The selected rows of [0, total) in chunks claimed from *counter. Warp 0
// claims two chunks ahead and stages the next one while the block copies
// the current one, so a chunk costs one barrier and no dependent index load.
template <int CPL, int kU>
__device__ __forceinline__ void claim_selected(const GatherArgs& a, unsigned* counter, int64_t total, int64_t jn,
                                               ChunkStage* st, unsigned* s_c) {
  const int64_t n_chunks = (total + kRowChunk - 1) / kRowChunk;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  unsigned ahead = 0;  // warp 0: the chunk claimed after the staged one
  if (warp == 0) {
    unsigned c = 0;
    if (lane == 0) {
      c = atomicAdd(counter, 1u);
      ahead = atomicAdd(counter, 1u);
    }
    c = __shfl_sync(0xffffffffu, c, 0);
    if (c < n_chunks) stage_chunk(a, c, total, jn, st[0]);
    cp_async_wait_all();
    if (lane == 0) s_c[0] = c;
  }
  __syncthreads();
  int buf = 0;
  unsigned c = s_c[0];
  while (c < n_chunks) {  // block-uniform
    if (warp == 0) {
      const unsigned nx = __shfl_sync(0xffffffffu, ahead, 0);
      if (nx < n_chunks) stage_chunk(a, nx, total, jn, st[buf ^ 1]);
      if (lane == 0) {
        s_c[buf ^ 1] = nx;
        ahead = atomicAdd(counter, 1u);
      }
    }
    copy_staged<CPL, kU>(a, st[buf], static_cast<int64_t>(c) * kRowChunk, jn);
    if (warp == 0) cp_async_wait_all();
    __syncthreads();  // the next chunk is staged; this one's stage may be reused
    buf ^= 1;
    c = s_c[buf];
  }
}

template <int CPL>
__global__ void __launch_bounds__(kGatherThreads, CPL >= 8 ? 2 : 4) gather_kernel(GatherArgs a) {
  pdl_trigger();
  constexpr int kU = CPL >= 4 ? 1 : 4 / CPL;
  __shared__ unsigned s_next;
  // The recent rows, while the selection runs.
  if (a.rp > 0) claim_recent<CPL, kU>(a, a.claim, a.n_slabs * a.rp, a.rp, &s_next);
  pdl_wait();  // the kept indices come from the selection kernel
  dev::gather_ids(a);
  // The selected (past) rows of every slab; handed out too, so that blocks on
  // SMs that HBM serves faster take more of them.
  const int64_t jn = a.budget - a.rp;
  __shared__ ChunkStage s_stage[2];
  __shared__ unsigned s_chunk[2];
  if (jn > 0) claim_selected<CPL, kU>(a, a.claim + 1, a.n_slabs * jn, jn, s_stage, s_chunk);
  // The last block out clears the counters for the next pass. Every pass
  // begins with a kernel launched without dependent-launch overlap, so the
  // next compaction cannot start before this one has finished.
  if (threadIdx.x == 0) {
    __threadfence();
    if (atomicAdd(a.claim + 2, 1u) == gridDim.x - 1) {
      a.claim[0] = 0;
      a.claim[1] = 0;
      a.claim[2] = 0;
      __threadfence();
    }
  }
}

template <int CPL>
cudaError_t dispatch(const GatherArgs& a, cudaStream_t st) {
  int per_sm = 0;
  cudaError_t e =
      cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_kernel<CPL>, kGatherThreads, 0);
  if (e != cudaSuccess) return e;
  per_sm = per_sm < 1 ? 1 : per_sm;
  return launch(gather_kernel<CPL>, a.num_sms * per_sm, kGatherThreads, 0, st, true, a);
}

}  // namespace

int gather_cpl(int row_bytes) {
  const int n_chunks = row_bytes / 16;
  return n_chunks <= 16 ? 1 : n_chunks <= 32 ? 2 : n_chunks <= 64 ? 4 : 8;
}

cudaError_t launch_gather(const GatherArgs& a, cudaStream_t st) {
  switch (gather_cpl(a.row_bytes)) {
    case 1: return dispatch<1>(a, st);
    case 2: return dispatch<2>(a, st);
    case 4: return dispatch<4>(a, st);
    default: return dispatch<8>(a, st);
  }
}

}  // namespace ipv
