// The shared index set (Sec. 3.1: K in R^{H x N x D}, compressed as
// K[:, I, :] with one I per layer): a token's TaR and VaN are those of its
// H x D key and value blocks read as single vectors,
//   s_TaR = -(sum_h k_h . m_{q,h}) / max(sqrt(sum_h |k_h|^2), eps),
//   s_VaN = sqrt(sum_h |v_h|^2),
// where m_{q,h} is head h's part of the block's recent-frame mean (built with
// the block norm). The scoring kernel leaves the per-head sums; this kernel
// adds them in head order. Elementwise over (layer, past row): a light pass
// over data the scoring kernel just wrote (L2-resident).
#include "ipv_common.cuh"

namespace ipv {
namespace {

__global__ void __launch_bounds__(256) combine_kernel(CombineArgs a) {
  pdl_trigger();
  pdl_wait();  // the partial sums come from the scoring kernel
  const int64_t total = a.n_layers * a.n_past;
  const int64_t step = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t g = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; g < total; g += step) {
    const int64_t l = g / a.n_past;
    const int64_t n = g - l * a.n_past;
    float dot = 0.0f, kk = 0.0f, vv = 0.0f;
    for (int h = 0; h < a.hs; ++h) {
      const int64_t i = (l * a.hs + h) * a.n_tokens + n;
      dot += a.dot[i];
      kk += a.kk[i];
      vv += a.vv[i];
    }
    a.tar[l * a.n_tokens + n] = -dot * rsqrtf(fmaxf(kk, kNormEps * kNormEps));
    a.van[l * a.n_tokens + n] = sqrtf(vv);  // NaN partials (no patch) stay NaN
  }
}

}  // namespace

cudaError_t launch_combine(const CombineArgs& a, cudaStream_t st) {
  const int64_t total = a.n_layers * a.n_past;
  int64_t blocks = (total + 255) / 256;
  const int64_t cap = static_cast<int64_t>(a.num_sms) * 8;
  blocks = blocks < cap ? blocks : cap;
  cudaError_t e = launch(combine_kernel, static_cast<unsigned>(blocks < 1 ? 1 : blocks), 256, 0, st,
                         true, a);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

}  // namespace ipv
