// Seeded synthetic KV-cache generator (device side). Test/bench harness only:
// it holds none of the compression method's arithmetic and is shared, as a
// source of input bytes, by the CUDA path's tests and the CPU oracle.
//
// Recipe (shapes and statistics of a 7B-class video MLLM's vision-token cache):
//   keys   per (slab, patch, dim): AR(1) across frames,
//          k_0 = e_0 / sqrt(1 - rho^2),  k_t = rho k_{t-1} + e_t,  e ~ N(0,1),
//          rho = rho[patch] (static or dynamic patch, chosen on the host);
//   values per token: v = (u / ||u||) * exp(sigma_l g),  u ~ N(0, I_D), where
//          g = beta_l S(t,i,j) + sqrt(1 - beta_l^2) z,  z ~ N(0,1), and S is a
//          smooth unit-variance field over each frame's grid (a sum of four
//          random low-frequency cosines drawn per (slab, frame)); sigma_l and
//          beta_l are per-layer (NULL arrays: sigma_l = sigma, beta_l = 0, g = z);
//   stored as bf16 (round to nearest even) or fp32.
// Random numbers: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel random
// numbers: as easy as 1, 2, 3", SC 2011), counter = (frame*p + patch, slab,
// purpose, dim/4), key = (seed low word, seed high word + stream); uniforms
// from the top 24 bits; normals by the Box-Muller transform.
#include <cuda_bf16.h>
#include <cuda_runtime.h>
#include <stdint.h>

namespace {

struct U4 {
  uint32_t a, b, c, d;
};

__device__ __forceinline__ U4 philox4x32_10(U4 x, uint32_t k0, uint32_t k1) {
#pragma unroll
  for (int round = 0; round < 10; ++round) {
    const uint32_t lo0 = 0xD2511F53u * x.a, hi0 = __umulhi(0xD2511F53u, x.a);
    const uint32_t lo1 = 0xCD9E8D57u * x.c, hi1 = __umulhi(0xCD9E8D57u, x.c);
    x = U4{hi1 ^ x.b ^ k0, lo1, hi0 ^ x.d ^ k1, lo0};
    k0 += 0x9E3779B9u;
    k1 += 0xBB67AE85u;
  }
  return x;
}

__device__ __forceinline__ float unit_open(uint32_t bits) {  // (0, 1)
  return ((bits >> 8) + 0.5f) * (1.0f / 16777216.0f);
}

__device__ __forceinline__ void four_normals(U4 r, float* z) {
  const float r0 = sqrtf(-2.0f * logf(unit_open(r.a)));
  const float r1 = sqrtf(-2.0f * logf(unit_open(r.c)));
  float s0, c0, s1, c1;
  sincospif(2.0f * unit_open(r.b), &s0, &c0);
  sincospif(2.0f * unit_open(r.d), &s1, &c1);
  z[0] = r0 * c0;
  z[1] = r0 * s0;
  z[2] = r1 * c1;
  z[3] = r1 * s1;
}

template <typename T>
__device__ __forceinline__ void store4(T* dst, const float* x);

template <>
__device__ __forceinline__ void store4<float>(float* dst, const float* x) {
  *reinterpret_cast<float4*>(dst) = make_float4(x[0], x[1], x[2], x[3]);
}

template <>
__device__ __forceinline__ void store4<__nv_bfloat16>(__nv_bfloat16* dst, const float* x) {
  __nv_bfloat162 lo = __floats2bfloat162_rn(x[0], x[1]);
  __nv_bfloat162 hi = __floats2bfloat162_rn(x[2], x[3]);
  uint2 w;
  w.x = *reinterpret_cast<uint32_t*>(&lo);
  w.y = *reinterpret_cast<uint32_t*>(&hi);
  *reinterpret_cast<uint2*>(dst) = w;
}

// One thread per (slab, patch, group of 4 dims); walks frames in order.
template <typename T>
__global__ void keys_kernel(T* k, int64_t n_slabs, int64_t cap, int D, int p, int frame0,
                            int n_frames, int64_t row0, const float* rho, float* state,
                            uint32_t key0, uint32_t key1, int64_t slab_base) {
  const int chunks = D / 4;
  const int64_t tid = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x;
  const int64_t total = n_slabs * p * chunks;
  if (tid >= total) return;
  const int c = static_cast<int>(tid % chunks);
  const int q = static_cast<int>((tid / chunks) % p);
  const int64_t s = tid / (static_cast<int64_t>(chunks) * p);
  const float rq = rho[q];
  const float init_scale = rsqrtf(fmaxf(1.0f - rq * rq, 1e-12f));
  float* st = state + (s * p + q) * D + 4 * c;
  float x[4] = {st[0], st[1], st[2], st[3]};
  for (int t = frame0; t < frame0 + n_frames; ++t) {
    const U4 ctr{static_cast<uint32_t>(t) * static_cast<uint32_t>(p) + q,
                 static_cast<uint32_t>(slab_base + s), 0u, static_cast<uint32_t>(c)};
    float z[4];
    four_normals(philox4x32_10(ctr, key0, key1), z);
#pragma unroll
    for (int i = 0; i < 4; ++i) x[i] = (t == 0) ? z[i] * init_scale : rq * x[i] + z[i];
    const int64_t row = row0 + static_cast<int64_t>(t - frame0) * p + q;
    store4<T>(k + (s * cap + row) * D + 4 * c, x);
  }
  st[0] = x[0];
  st[1] = x[1];
  st[2] = x[2];
  st[3] = x[3];
}

// One warp per token row: u ~ N(0, I_D) normalised, scaled by a lognormal.
// Smooth unit-variance field over a frame's gh x gw grid at patch (i, j):
// sum over a < 4 of sqrt(1/2) cos(2 pi (u_a i / gh + v_a j / gw + phi_a)), with
// u_a, v_a in {0, 1, 2} and phi_a uniform, drawn once per (slab, frame).
__device__ float frame_field(uint32_t frame, uint32_t slab, int i, int j, int gh, int gw,
                             uint32_t key0, uint32_t key1) {
  const U4 w = philox4x32_10(U4{frame, slab, 3u, 0u}, key0, key1);
  const U4 ph = philox4x32_10(U4{frame, slab, 4u, 0u}, key0, key1);
  const uint32_t ws[4] = {w.a, w.b, w.c, w.d};
  const uint32_t phs[4] = {ph.a, ph.b, ph.c, ph.d};
  float acc = 0.0f;
#pragma unroll
  for (int a = 0; a < 4; ++a) {
    const float u = static_cast<float>(ws[a] % 3u);
    const float vv = static_cast<float>((ws[a] / 3u) % 3u);
    const float x = u * static_cast<float>(i) / static_cast<float>(gh) +
                    vv * static_cast<float>(j) / static_cast<float>(gw) + unit_open(phs[a]);
    acc += 0.70710678f * cospif(2.0f * x);
  }
  return acc;
}

struct ValueParams {
  const float* layer_sigma;  // [n_layers] or NULL
  const float* layer_beta;   // [n_layers] or NULL
  int n_layers, n_kv_heads, grid_w;
};

template <typename T>
__global__ void values_kernel(T* v, int64_t n_slabs, int64_t cap, int D, int p, int frame0,
                              int n_frames, int64_t row0, float sigma, uint32_t key0,
                              uint32_t key1, int64_t slab_base, ValueParams vp) {
  const int lane = threadIdx.x & 31;
  const int64_t warp = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
  const int64_t rows = static_cast<int64_t>(n_frames) * p;
  if (warp >= n_slabs * rows) return;
  const int64_t s = warp / rows;
  const int64_t i = warp % rows;
  const uint32_t token = static_cast<uint32_t>(frame0) * static_cast<uint32_t>(p) +
                         static_cast<uint32_t>(i);
  const uint32_t slab = static_cast<uint32_t>(slab_base + s);
  const int chunks = D / 4;
  float u[16][4];  // D <= 2048
  float ss = 0.0f;
  for (int j = 0; j < 16; ++j) {
    const int c = lane + 32 * j;
    if (c < chunks) {
      four_normals(philox4x32_10(U4{token, slab, 1u, static_cast<uint32_t>(c)}, key0, key1), u[j]);
      ss += u[j][0] * u[j][0] + u[j][1] * u[j][1] + u[j][2] * u[j][2] + u[j][3] * u[j][3];
    }
  }
  for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
  float zm[4];
  four_normals(philox4x32_10(U4{token, slab, 2u, 0u}, key0, key1), zm);
  float sig = sigma, g = zm[0];
  if (vp.layer_sigma) {
    const int layer = static_cast<int>((slab / static_cast<uint32_t>(vp.n_kv_heads)) %
                                       static_cast<uint32_t>(vp.n_layers));
    sig = vp.layer_sigma[layer];
    const float beta = vp.layer_beta[layer];
    if (beta != 0.0f) {
      const int q = static_cast<int>(token % static_cast<uint32_t>(p));
      const float field = frame_field(token / static_cast<uint32_t>(p), slab, q / vp.grid_w,
                                      q % vp.grid_w, p / vp.grid_w, vp.grid_w, key0, key1);
      g = beta * field + sqrtf(1.0f - beta * beta) * zm[0];
    }
  }
  const float scale = expf(sig * g) / sqrtf(ss);
  T* row = v + (s * cap + row0 + i) * D;
  for (int j = 0; j < 16; ++j) {
    const int c = lane + 32 * j;
    if (c < chunks) {
      float x[4] = {u[j][0] * scale, u[j][1] * scale, u[j][2] * scale, u[j][3] * scale};
      store4<T>(row + 4 * c, x);
    }
  }
}

template <typename T>
cudaError_t launch(void* k, void* v, int64_t n_slabs, int64_t cap, int D, int p, int frame0,
                   int n_frames, int64_t row0, const float* rho, float* state, float sigma,
                   uint64_t seed, uint32_t stream_id, int64_t slab_base, ValueParams vp,
                   cudaStream_t st) {
  const uint32_t key0 = static_cast<uint32_t>(seed);
  const uint32_t key1 = static_cast<uint32_t>(seed >> 32) + stream_id;
  const int64_t kthreads = n_slabs * p * (D / 4);
  keys_kernel<T><<<static_cast<unsigned>((kthreads + 255) / 256), 256, 0, st>>>(
      static_cast<T*>(k), n_slabs, cap, D, p, frame0, n_frames, row0, rho, state, key0, key1,
      slab_base);
  const int64_t vwarps = n_slabs * n_frames * static_cast<int64_t>(p);
  values_kernel<T><<<static_cast<unsigned>((vwarps * 32 + 255) / 256), 256, 0, st>>>(
      static_cast<T*>(v), n_slabs, cap, D, p, frame0, n_frames, row0, sigma, key0, key1,
      slab_base, vp);
  return cudaGetLastError();
}

}  // namespace

extern "C" {

// Writes frames [frame0, frame0 + n_frames) of every slab into rows
// row0 + (t - frame0) * p + patch of k and v ([n_slabs][cap][D], bf16 or
// fp32). rho: device [p]. state: device fp32 [n_slabs][p][D] holding the last
// key of each AR(1) chain (read unless frame0 == 0, always written back).
// layer_sigma, layer_beta: device fp32 [n_layers] per-layer value spread and
// spatial weight (both NULL: sigma for every layer, no spatial field); slab
// s + slab_base belongs to layer ((s + slab_base) / n_kv_heads) mod n_layers.
// Returns 0 or a cudaError_t value; 1000 for bad arguments.
int synth_fill(void* k, void* v, int is_bf16, int64_t n_slabs, int64_t cap, int D, int p,
               int frame0, int n_frames, int64_t row0, const float* rho, float* state,
               float sigma, uint64_t seed, uint32_t stream_id, int64_t slab_base,
               const float* layer_sigma, const float* layer_beta, int n_layers, int n_kv_heads,
               int grid_w, void* stream) {
  if (!k || !v || !rho || !state || n_slabs <= 0 || D <= 0 || D % 4 != 0 || D > 2048 ||
      p <= 0 || frame0 < 0 || n_frames <= 0 || row0 < 0 ||
      row0 + static_cast<int64_t>(n_frames) * p > cap)
    return 1000;
  if ((layer_sigma == nullptr) != (layer_beta == nullptr)) return 1000;
  if (layer_sigma && (n_layers <= 0 || n_kv_heads <= 0 || grid_w <= 0 || p % grid_w != 0))
    return 1000;
  const ValueParams vp{layer_sigma, layer_beta, n_layers, n_kv_heads, grid_w};
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (is_bf16)
    return launch<__nv_bfloat16>(k, v, n_slabs, cap, D, p, frame0, n_frames, row0, rho, state,
                                 sigma, seed, stream_id, slab_base, vp, st);
  return launch<float>(k, v, n_slabs, cap, D, p, frame0, n_frames, row0, rho, state, sigma,
                       seed, stream_id, slab_base, vp, st);
}

}  // extern "C"
