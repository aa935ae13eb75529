// Step (iv) of the compression pass: compaction of the kept rows.
//
// InfiniPot-V Sec. 3.1 / Algorithm 2 last step: K~ = K[:, J, :], V~ = V[:, J, :]
// with J ascending, i.e. dst row j of a slab is src row kept[j], bytes
// unchanged. The destination is the other half of the ping-pong cache, so the
// copy has no read/write hazards and the source stays intact.
//
// Pure data movement (HBM-bound): a half-warp moves one 16-byte-chunked K row
// and the matching V row; the flattened (slab, j) space is strided over the
// whole grid with several rows in flight per half-warp. The recent frames
// (always kept, always the last rp kept rows) are copied before the kernel
// waits for the selection, overlapping it. Patch and frame ids travel with
// their rows, copied by a separate coalesced loop.
#include "pass_device.cuh"

namespace ipv {
namespace {

template <int CPL>
__global__ void __launch_bounds__(512, CPL >= 8 ? 1 : 2) gather_kernel(GatherArgs a) {
  pdl_trigger();
  constexpr int kU = CPL >= 4 ? 1 : 4 / CPL;
  const int64_t n_hw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 4;
  const int64_t hw = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 4;
  // The recent frames are always kept, as the last rp kept rows: copy them
  // while the selection is still running (it leaves HBM idle).
  if (a.rp > 0) dev::gather_range<CPL, kU, false, false, true>(a, 0, a.n_slabs * a.rp, hw, n_hw, a.rp);
  pdl_wait();  // the kept indices come from the selection kernel
  dev::gather_ids(a);
  const int64_t jn = a.budget - a.rp;  // the selected (past) rows of every slab
  dev::gather_range<CPL, kU, false, false>(a, 0, a.n_slabs * jn, hw, n_hw, jn);
}

template <int CPL>
cudaError_t dispatch(const GatherArgs& a, cudaStream_t st) {
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_kernel<CPL>, 512, 0);
  if (e != cudaSuccess) return e;
  per_sm = per_sm < 1 ? 1 : per_sm;
  return launch(gather_kernel<CPL>, a.num_sms * per_sm, 512, 0, st, true, a);
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
