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
// the same way after the wait. Patch and frame ids travel with their rows,
// copied by a separate coalesced loop.
#include "pass_device.cuh"

namespace ipv {
namespace {

constexpr int kGatherThreads = 256;   // 64 registers: one block fits beside a selection block
constexpr int64_t kRowChunk = 128;    // rows per claim

// Copies the chunks of [0, total) rows (kRowChunk each) that the block claims
// from *counter, the next claim in flight while a chunk is copied.
template <int CPL, int kU, bool FIXED>
__device__ __forceinline__ void claim_rows(const GatherArgs& a, unsigned* counter, int64_t total, int64_t jn,
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
    dev::gather_range<CPL, kU, false, FIXED>(a, b0, min(total, b0 + kRowChunk), threadIdx.x >> 4,
                                                    blockDim.x >> 4, jn);
    __syncthreads();  // every thread has read *s_next
    if (threadIdx.x == 0) *s_next = nxt;
    __syncthreads();
    c = *s_next;
  }
}

template <int CPL>
__global__ void __launch_bounds__(kGatherThreads, CPL >= 8 ? 2 : 4) gather_kernel(GatherArgs a) {
  pdl_trigger();
  constexpr int kU = CPL >= 4 ? 1 : 4 / CPL;
  __shared__ unsigned s_next;
  // The recent rows, while the selection runs.
  if (a.rp > 0) claim_rows<CPL, kU, true>(a, a.claim, a.n_slabs * a.rp, a.rp, &s_next);
  pdl_wait();  // the kept indices come from the selection kernel
  dev::gather_ids(a);
  // The selected (past) rows of every slab; handed out too, so that blocks on
  // SMs that HBM serves faster take more of them.
  const int64_t jn = a.budget - a.rp;
  claim_rows<CPL, kU, false>(a, a.claim + 1, a.n_slabs * jn, jn, &s_next);
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
