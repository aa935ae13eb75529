// Algorithm 1's accumulate step for a streaming cache: whole new frames are
// appended behind the rows already cached in every slab, with their patch ids
// (the frame-grid position, row offset mod p) and frame ids (continuing from
// the last cached row's frame, numbered on the device so that a captured CUDA
// graph can replay the step). The appended rows are the next pass's recent
// frames and most recent past rows, so they are stored with ordinary (L2-
// allocating) stores. HBM-bound copy: a half-warp moves one K row and the
// matching V row in 16-byte chunks.
#include "ipv_common.cuh"

namespace ipv {
namespace {

template <int CPL>
__global__ void __launch_bounds__(512) append_kernel(AppendArgs a) {
  const int lane = threadIdx.x & 15;
  const int n_chunks = a.row_bytes / 16;
  const int64_t n_hw = (static_cast<int64_t>(gridDim.x) * blockDim.x) >> 4;
  const int64_t total = a.n_slabs * a.n_new;
  const char* ks = static_cast<const char*>(a.k_new);
  const char* vs = static_cast<const char*>(a.v_new);
  char* kd = static_cast<char*>(a.k_dst);
  char* vd = static_cast<char*>(a.v_dst);
  for (int64_t g = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 4; g < total;
       g += n_hw) {
    const int64_t s = g / a.n_new;
    const int64_t t = g - s * a.n_new;          // row within the new frames
    const int64_t src = g * a.row_bytes;
    const int64_t dst = (s * a.cap + a.row0 + t) * a.row_bytes;
    uint4 kr[CPL], vr[CPL];
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      const int ch = lane + 16 * c;
      kr[c] = ch < n_chunks ? ld_stream(ks + src + ch * 16) : make_uint4(0, 0, 0, 0);
      vr[c] = ch < n_chunks ? ld_stream(vs + src + ch * 16) : make_uint4(0, 0, 0, 0);
    }
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      const int ch = lane + 16 * c;
      if (ch < n_chunks) {
        *reinterpret_cast<uint4*>(kd + dst + ch * 16) = kr[c];
        *reinterpret_cast<uint4*>(vd + dst + ch * 16) = vr[c];
      }
    }
    if (lane == 0 && a.pid) a.pid[s * a.cap + a.row0 + t] = static_cast<uint16_t>(t % a.p);
    if (lane == 1 && a.fid) {
      // The frame after the last cached row's frame (first_frame for an empty slab).
      const uint32_t base = a.row0 > 0 ? a.fid[s * a.cap + a.row0 - 1] + 1u : a.first_frame;
      a.fid[s * a.cap + a.row0 + t] = base + static_cast<uint32_t>(t / a.p);
    }
  }
}

template <int CPL>
cudaError_t dispatch(const AppendArgs& a, cudaStream_t st) {
  const int64_t rows = a.n_slabs * a.n_new;
  int64_t blocks = (rows * 16 + 511) / 512;
  const int64_t cap = static_cast<int64_t>(a.num_sms) * 4;
  blocks = blocks < cap ? blocks : cap;
  append_kernel<CPL><<<static_cast<unsigned>(blocks < 1 ? 1 : blocks), 512, 0, st>>>(a);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_append(const AppendArgs& a, cudaStream_t st) {
  switch (gather_cpl(a.row_bytes)) {
    case 1: return dispatch<1>(a, st);
    case 2: return dispatch<2>(a, st);
    case 4: return dispatch<4>(a, st);
    default: return dispatch<8>(a, st);
  }
}

}  // namespace ipv
