// Steps (i) and (ii) of the compression pass: TaR and VaN scores.
//
// TaR (InfiniPot-V Sec. 3.1, Eq. tar) averages r cosines per past token:
//   s_TaR(n) = -(1/r) sum_{t'} k_n.k_{t'} / (max|k_n|,eps) (max|k_{t'}|,eps),
// with k_{t'} the key at the same patch q(n) in recent frame t'. Pulling the
// past-token factor out of the sum gives the exact regrouping
//   s_TaR(n) = -(k_n . m_q) / max|k_n|,eps,   m_q = (1/r) sum_{t'} k_{t'} / max|k_{t'}|,eps,
// so each key row is read once: recent_mean_kernel builds m_q per (slab,
// patch) from the r recent rows, score_kernel streams every past K and V row
// once and finishes both scores (VaN, Sec. 3.2: s_VaN = |v|_2).
//
// Both kernels are HBM-bound scans (about 2 flops per byte). A row (head_dim
// elements, a multiple of 16 bytes) is read by a small lane group with
// 16-byte loads; sums are fp32 lane partials combined by a shuffle tree.
#include "pass_device.cuh"

namespace ipv {
namespace {

constexpr int kScoreThreads = 768;
constexpr int kPrefetchRows = 256;  // rows of K and of V fetched into L2 before the wait

// m_q for 32/LPR patches per warp, patches flattened over (slab, q); with
// VIRT a "slab" is a layer whose a.hs heads form one token block.
template <typename T, int LPR, int CPL, bool VIRT>
__global__ void __launch_bounds__(128) recent_mean_kernel(ScoreArgs a) {
  pdl_trigger();
  constexpr int RPW = 32 / LPR;
  const int grp = (threadIdx.x & 31) / LPR;
  const int64_t warp = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
  const int64_t col = warp * RPW + grp;
  const bool col_ok = col < a.n_slabs * a.p;
  const int64_t s = col_ok ? col / a.p : 0;
  const int q = col_ok ? static_cast<int>(col - s * a.p) : 0;
  dev::mean_group<T, LPR, CPL, VIRT>(a, s, q, col_ok);
}

// Streams the past rows. Block b owns an equal contiguous share of the
// flattened (slab, past row) space; for each slab its share touches, the
// slab's m table is staged in shared memory with rows padded to D+4 floats
// (SMEM_M), or read through L1/L2.
template <typename T, int LPR, int CPL, bool SMEM_M>
__global__ void __launch_bounds__(kScoreThreads, 1) score_kernel(ScoreArgs a) {
  pdl_trigger();
  constexpr int kU = CPL >= 4 ? 1 : 4 / CPL;
  extern __shared__ float4 sm_m4[];
  const int lane = threadIdx.x & 31;
  const int warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  const int ms = SMEM_M ? a.D + 4 : a.D;  // m row stride (floats)
  const int64_t n_past = a.n_tokens - static_cast<int64_t>(a.r) * a.p;
  const int64_t total = a.n_slabs * n_past;
  const int64_t end = total * (blockIdx.x + 1) / gridDim.x;
  int64_t pos = total * blockIdx.x / gridDim.x;
  if (threadIdx.x == 0 && pos < end) {
    // K and V do not depend on the recent-frame mean: while its last blocks
    // run, the first rows of this block's share are fetched into L2.
    const int64_t s0 = pos / n_past;
    const int64_t lo0 = pos - s0 * n_past;
    const uint32_t bytes = static_cast<uint32_t>(min(min(n_past - lo0, end - pos), static_cast<int64_t>(kPrefetchRows)) *
                                                 a.D * static_cast<int>(sizeof(T)));
    const int64_t off = (s0 * a.cap + lo0) * a.D * static_cast<int64_t>(sizeof(T));
    prefetch_l2(static_cast<const char*>(a.k) + off, bytes);
    prefetch_l2(static_cast<const char*>(a.v) + off, bytes);
  }
  pdl_wait();  // m comes from the recent-frame mean kernel
  while (pos < end) {  // block-uniform
    const int64_t s = pos / n_past;
    const int lo = static_cast<int>(pos - s * n_past);
    const int hi = static_cast<int>(min(n_past, static_cast<int64_t>(lo) + (end - pos)));
    const float* m_slab = a.m + s * a.p * static_cast<int64_t>(a.D);
    if (SMEM_M) {
      __syncthreads();  // the previous slab's table is no longer read
      // Every copy of the table is in flight at once: a row per warp and
      // iteration with plain loads would take a dependent L2 round trip per
      // row while the other SMs keep HBM saturated.
      const int d4 = a.D / 4;
      for (int q = warp; q < a.p; q += n_warps) {
        const float4* src = reinterpret_cast<const float4*>(m_slab + static_cast<int64_t>(q) * a.D);
        float4* dst = sm_m4 + q * (ms / 4);
        for (int j = lane; j < d4; j += 32) cp_async16(dst + j, src + j);
      }
      cp_async_wait_all();
      __syncthreads();
      dev::score_segment<T, LPR, CPL, kU, dev::kMSmem>(a, s, lo, hi,
                                                       reinterpret_cast<const float*>(sm_m4), ms);
    } else {
      dev::score_segment<T, LPR, CPL, kU, dev::kMGlobalRO>(a, s, lo, hi, m_slab, ms);
    }
    pos += hi - lo;
  }
}

constexpr size_t kScoreSmemLimit = 200 * 1024;

template <typename T, int LPR, int CPL>
cudaError_t dispatch_score(const ScoreArgs& a, cudaStream_t st) {
  const size_t smem = score_smem_bytes(a.p, a.D);
  int per_sm = 0;
  cudaError_t e;
  if (smem > 0) {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<T, LPR, CPL, true>,
                                                      kScoreThreads, smem);
    if (e != cudaSuccess) return e;
    per_sm = per_sm < 1 ? 1 : per_sm;
    e = launch(score_kernel<T, LPR, CPL, true>, a.num_sms * per_sm, kScoreThreads, smem, st, true, a);
    if (e != cudaSuccess) return e;
  } else {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<T, LPR, CPL, false>,
                                                      kScoreThreads, 0);
    if (e != cudaSuccess) return e;
    per_sm = per_sm < 1 ? 1 : per_sm;
    e = launch(score_kernel<T, LPR, CPL, false>, a.num_sms * per_sm, kScoreThreads, 0, st, true, a);
    if (e != cudaSuccess) return e;
  }
  return cudaGetLastError();
}

template <typename T, int LPR, int CPL>
cudaError_t dispatch_mean(const ScoreArgs& a, cudaStream_t st) {
  const int64_t warps = (a.n_slabs * a.p + (32 / LPR) - 1) / (32 / LPR);
  const unsigned grid = static_cast<unsigned>((warps * 32 + 127) / 128);
  if (a.hs > 1)
    recent_mean_kernel<T, LPR, CPL, true><<<grid, 128, 0, st>>>(a);
  else
    recent_mean_kernel<T, LPR, CPL, false><<<grid, 128, 0, st>>>(a);
  return cudaGetLastError();
}

template <typename T, int LPR, int CPL>
cudaError_t set_smem_attr() {
  return cudaFuncSetAttribute(score_kernel<T, LPR, CPL, true>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(kScoreSmemLimit));
}

template <typename T>
cudaError_t prepare_t() {
  cudaError_t e;
  if ((e = set_smem_attr<T, 4, 1>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<T, 4, 2>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<T, 4, 4>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<T, 8, 4>()) != cudaSuccess) return e;
  if ((e = set_smem_attr<T, 16, 4>()) != cudaSuccess) return e;
  return set_smem_attr<T, 16, 8>();
}

template <typename T, bool MEAN>
cudaError_t dispatch_t(const ScoreArgs& a, cudaStream_t st) {
  // The recent-frame mean of the shared index set reads hs head-rows per token.
  const int width = MEAN && a.hs > 1 ? a.D * a.hs : a.D;
  switch (row_shape(width, a.is_bf16)) {
    case 41: return MEAN ? dispatch_mean<T, 4, 1>(a, st) : dispatch_score<T, 4, 1>(a, st);
    case 42: return MEAN ? dispatch_mean<T, 4, 2>(a, st) : dispatch_score<T, 4, 2>(a, st);
    case 44: return MEAN ? dispatch_mean<T, 4, 4>(a, st) : dispatch_score<T, 4, 4>(a, st);
    case 84: return MEAN ? dispatch_mean<T, 8, 4>(a, st) : dispatch_score<T, 8, 4>(a, st);
    case 164: return MEAN ? dispatch_mean<T, 16, 4>(a, st) : dispatch_score<T, 16, 4>(a, st);
    default: return MEAN ? dispatch_mean<T, 16, 8>(a, st) : dispatch_score<T, 16, 8>(a, st);
  }
}

}  // namespace

int row_shape(int D, int is_bf16) {
  const int n_chunks = D * (is_bf16 ? 2 : 4) / 16;
  return n_chunks <= 4 ? 41 : n_chunks <= 8 ? 42 : n_chunks <= 16 ? 44 : n_chunks <= 32 ? 84
         : n_chunks <= 64 ? 164 : 168;
}

size_t score_smem_bytes(int p, int D) {
  const size_t b = static_cast<size_t>(p) * (D + 4) * sizeof(float);
  return b <= kScoreSmemLimit ? b : 0;  // 0: m is read through L1/L2 instead
}

cudaError_t score_prepare(int, int) {
  cudaError_t e = prepare_t<uint16_t>();
  if (e == cudaSuccess) e = prepare_t<float>();
  return e;
}

cudaError_t launch_recent_mean(const ScoreArgs& a, cudaStream_t st) {
  return a.is_bf16 ? dispatch_t<uint16_t, true>(a, st) : dispatch_t<float, true>(a, st);
}

cudaError_t launch_score(const ScoreArgs& a, cudaStream_t st) {
  return a.is_bf16 ? dispatch_t<uint16_t, false>(a, st) : dispatch_t<float, false>(a, st);
}

}  // namespace ipv
