// Step (iv) of the compression pass: compaction of the kept rows.
//
// InfiniPot-V Sec. 3.1 / Algorithm 2 last step: K~ = K[:, J, :], V~ = V[:, J, :]
// with J ascending, i.e. dst row j of a slab is src row kept[j], bytes
// unchanged. The destination is the other half of the ping-pong cache, so the
// copy has no read/write hazards and the source stays intact.
//
// Pure data movement (HBM-bound): a half-warp moves one 16-byte-chunked K row
// and the matching V row; the flattened (slab, j) space is strided over the
// whole grid with several rows in flight per half-warp. Patch ids travel with
// their rows.
#include "ipv_common.cuh"

namespace ipv {
namespace {

template <int CPL>
__global__ void __launch_bounds__(512, 2) gather_kernel(GatherArgs a) {
  constexpr int kUnroll = CPL >= 4 ? 1 : 4 / CPL;
  const int lane = threadIdx.x & 15;
  const int64_t n_hw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 4;
  const int64_t hw = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 4;
  const int64_t total = a.n_slabs * a.budget;
  const int n_chunks = a.row_bytes / 16;
  const char* ks = static_cast<const char*>(a.k_src);
  const char* vs = static_cast<const char*>(a.v_src);
  char* kd = static_cast<char*>(a.k_dst);
  char* vd = static_cast<char*>(a.v_dst);

  for (int64_t g0 = hw; g0 < total; g0 += n_hw * kUnroll) {
    uint4 kr[kUnroll][CPL], vr[kUnroll][CPL];
    int64_t dst_off[kUnroll];
    int src_n[kUnroll];
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      const int64_t g = g0 + u * n_hw;
      int n = -1;
      int64_t s = 0, j = 0;
      if (g < total) {
        s = g / a.budget;
        j = g - s * a.budget;
        n = a.kept[g];
        if (n >= a.cap) n = -1;  // never produced by the selection; ignore
      }
      src_n[u] = n;
      dst_off[u] = (s * a.cap + j) * a.row_bytes;
      const int64_t src_off = (s * a.cap + (n < 0 ? 0 : n)) * a.row_bytes;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        const bool ld = n >= 0 && ch < n_chunks;
        kr[u][c] = ld ? ld_stream(ks + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
        vr[u][c] = ld ? ld_stream(vs + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int u = 0; u < kUnroll; ++u) {
      if (src_n[u] < 0) continue;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        if (ch < n_chunks) {
          st_stream(kd + dst_off[u] + ch * 16, kr[u][c]);
          st_stream(vd + dst_off[u] + ch * 16, vr[u][c]);
        }
      }
      if (a.pid_dst && lane == 0) {
        const int64_t g = g0 + u * n_hw;
        const int64_t s = g / a.budget;
        const int64_t j = g - s * a.budget;
        a.pid_dst[s * a.cap + j] = a.pid_src ? a.pid_src[s * a.cap + src_n[u]]
                                             : static_cast<uint16_t>(src_n[u] % a.p);
      }
    }
  }
}

template <int CPL>
cudaError_t dispatch(const GatherArgs& a, cudaStream_t st) {
  int per_sm = 0;
  cudaError_t e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gather_kernel<CPL>, 512, 0);
  if (e != cudaSuccess) return e;
  per_sm = per_sm < 1 ? 1 : per_sm;
  gather_kernel<CPL><<<a.num_sms * per_sm, 512, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gather(const GatherArgs& a, cudaStream_t st) {
  const int n_chunks = a.row_bytes / 16;
  const int cpl = n_chunks <= 16 ? 1 : n_chunks <= 32 ? 2 : n_chunks <= 64 ? 4 : 8;
  switch (cpl) {
    case 1: return dispatch<1>(a, st);
    case 2: return dispatch<2>(a, st);
    case 4: return dispatch<4>(a, st);
    default: return dispatch<8>(a, st);
  }
}

}  // namespace ipv
