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
// elements, a multiple of 16 bytes) is read by a half-warp with 16-byte
// loads; sums are fp32 lane partials combined by a shuffle tree.
#include "ipv_common.cuh"

namespace ipv {
namespace {

__device__ __forceinline__ unsigned halfwarp_mask() {
  return (threadIdx.x & 16) ? 0xFFFF0000u : 0x0000FFFFu;
}

__device__ __forceinline__ float hsum(unsigned mask, float x) {
  x += __shfl_xor_sync(mask, x, 8);
  x += __shfl_xor_sync(mask, x, 4);
  x += __shfl_xor_sync(mask, x, 2);
  x += __shfl_xor_sync(mask, x, 1);
  return x;
}

// One half-warp per (slab, patch): m_q = (1/r) sum_t' k_t'/max(|k_t'|, eps).
template <typename T, int CPL>
__global__ void __launch_bounds__(256) recent_mean_kernel(ScoreArgs a) {
  constexpr int E = Chunk<T>::kElems;
  constexpr int kBatch = 4;
  const int lane = threadIdx.x & 15;
  const unsigned mask = halfwarp_mask();
  const int64_t col = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 4;
  if (col >= a.n_slabs * a.p) return;  // uniform per half-warp
  const int64_t s = col / a.p;
  const int q = static_cast<int>(col - s * a.p);
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int64_t n_past = a.n_tokens - static_cast<int64_t>(a.r) * a.p;
  const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;

  float acc[CPL][E];
#pragma unroll
  for (int c = 0; c < CPL; ++c)
#pragma unroll
    for (int e = 0; e < E; ++e) acc[c][e] = 0.0f;

  for (int t0 = 0; t0 < a.r; t0 += kBatch) {
    uint4 raw[kBatch][CPL];
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      const int64_t n = n_past + static_cast<int64_t>(t0 + b) * a.p + q;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        raw[b][c] = (t0 + b < a.r && ch < n_chunks) ? ld_stream(kslab + n * row_bytes + ch * 16)
                                                    : make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      if (t0 + b >= a.r) break;  // uniform per half-warp
      float x[CPL][E];
      float kk = 0.0f;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        Chunk<T>::widen(raw[b][c], x[c]);
#pragma unroll
        for (int e = 0; e < E; ++e) kk = fmaf(x[c][e], x[c][e], kk);
      }
      kk = hsum(mask, kk);
      const float inv = 1.0f / fmaxf(sqrtf(kk), kNormEps);
#pragma unroll
      for (int c = 0; c < CPL; ++c)
#pragma unroll
        for (int e = 0; e < E; ++e) acc[c][e] = fmaf(x[c][e], inv, acc[c][e]);
    }
  }
  const float rf = static_cast<float>(a.r);
  float* mrow = a.m + (s * a.p + q) * static_cast<int64_t>(a.D);
#pragma unroll
  for (int c = 0; c < CPL; ++c) {
    const int ch = lane + 16 * c;
    if (ch < n_chunks) {
#pragma unroll
      for (int e = 0; e < E; e += 4)
        *reinterpret_cast<float4*>(mrow + ch * E + e) =
            make_float4(acc[c][e] / rf, acc[c][e + 1] / rf, acc[c][e + 2] / rf, acc[c][e + 3] / rf);
    }
  }
  if (a.zero_recent && lane == 0) {
    for (int t = 0; t < a.r; ++t) {
      const int64_t n = n_past + static_cast<int64_t>(t) * a.p + q;
      a.tar[s * a.n_tokens + n] = 0.0f;
      a.van[s * a.n_tokens + n] = 0.0f;
    }
  }
}

// Streams the past rows. Block b owns an equal contiguous share of the
// flattened (slab, past row) space; for each slab its share touches, the
// slab's m table ([p][D] fp32) is staged in shared memory (SMEM_M) or read
// through L2. Half-warp h takes rows h, h+32, ... of the share, kUnroll rows
// in flight.
template <typename T, int CPL, bool SMEM_M>
__global__ void __launch_bounds__(512, 1) score_kernel(ScoreArgs a) {
  constexpr int E = Chunk<T>::kElems;
  constexpr int kUnroll = CPL >= 4 ? 1 : 4 / CPL;
  extern __shared__ float4 sm_m4[];
  const float* sm_m = reinterpret_cast<const float*>(sm_m4);
  const int lane = threadIdx.x & 15;
  const int hw = threadIdx.x >> 4;
  const int n_hw = blockDim.x >> 4;
  const unsigned mask = halfwarp_mask();
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int64_t n_past = a.n_tokens - static_cast<int64_t>(a.r) * a.p;
  const int64_t total = a.n_slabs * n_past;
  const int64_t end = total * (blockIdx.x + 1) / gridDim.x;
  int64_t pos = total * blockIdx.x / gridDim.x;

  while (pos < end) {  // block-uniform
    const int64_t s = pos / n_past;
    const int64_t lo = pos - s * n_past;
    const int64_t hi = min(n_past, lo + (end - pos));
    const float* m_slab = a.m + s * a.p * static_cast<int64_t>(a.D);
    if (SMEM_M) {
      __syncthreads();
      const float4* src = reinterpret_cast<const float4*>(m_slab);
      const int n4 = a.p * a.D / 4;
      for (int i = threadIdx.x; i < n4; i += blockDim.x) sm_m4[i] = src[i];
      __syncthreads();
    }
    const float* mtab = SMEM_M ? sm_m : m_slab;
    const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;
    const char* vslab = static_cast<const char*>(a.v) + s * a.cap * row_bytes;
    const uint16_t* pid = a.patch_id ? a.patch_id + s * a.cap : nullptr;
    float* tar = a.tar + s * a.n_tokens;
    float* van = a.van + s * a.n_tokens;

    for (int64_t n0 = lo + hw; n0 < hi; n0 += static_cast<int64_t>(n_hw) * kUnroll) {
      uint4 kr[kUnroll][CPL], vr[kUnroll][CPL];
      int q[kUnroll];
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t n = n0 + static_cast<int64_t>(u) * n_hw;
        const bool ok = n < hi;
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
          const int ch = lane + 16 * c;
          const bool ld = ok && ch < n_chunks;
          kr[u][c] = ld ? ld_stream(kslab + n * row_bytes + ch * 16) : make_uint4(0, 0, 0, 0);
          vr[u][c] = ld ? ld_stream(vslab + n * row_bytes + ch * 16) : make_uint4(0, 0, 0, 0);
        }
        q[u] = ok ? (pid ? static_cast<int>(pid[n]) : static_cast<int>(n % a.p)) : 0;
      }
#pragma unroll
      for (int u = 0; u < kUnroll; ++u) {
        const int64_t n = n0 + static_cast<int64_t>(u) * n_hw;
        if (n >= hi) break;  // uniform per half-warp
        const bool q_ok = q[u] < a.p;
        const float* mq = mtab + static_cast<int64_t>(q_ok ? q[u] : 0) * a.D;
        float dot = 0.0f, kk = 0.0f, vv = 0.0f;
#pragma unroll
        for (int c = 0; c < CPL; ++c) {
          const int ch = lane + 16 * c;
          float kx[E], vx[E];
          Chunk<T>::widen(kr[u][c], kx);
          Chunk<T>::widen(vr[u][c], vx);
          if (ch < n_chunks) {
#pragma unroll
            for (int e = 0; e < E; e += 4) {
              const float4 mv = *reinterpret_cast<const float4*>(mq + ch * E + e);
              dot = fmaf(kx[e], mv.x, dot);
              dot = fmaf(kx[e + 1], mv.y, dot);
              dot = fmaf(kx[e + 2], mv.z, dot);
              dot = fmaf(kx[e + 3], mv.w, dot);
            }
          }
#pragma unroll
          for (int e = 0; e < E; ++e) {
            kk = fmaf(kx[e], kx[e], kk);
            vv = fmaf(vx[e], vx[e], vv);
          }
        }
        dot = hsum(mask, dot);
        kk = hsum(mask, kk);
        vv = hsum(mask, vv);
        if (lane == 0) {
          // A patch id outside [0, p) has no recent-frame partner: NaN scores
          // rank below every number, so such a token is never preferred.
          tar[n] = q_ok ? -dot / fmaxf(sqrtf(kk), kNormEps) : __int_as_float(0x7fc00000);
          van[n] = q_ok ? sqrtf(vv) : __int_as_float(0x7fc00000);
        }
      }
    }
    pos += hi - lo;
  }
}

constexpr size_t kScoreSmemLimit = 200 * 1024;

template <typename T, int CPL>
cudaError_t dispatch_score(const ScoreArgs& a, cudaStream_t st) {
  const size_t smem = score_smem_bytes(a.p, a.D);
  int per_sm = 0;
  cudaError_t e;
  if (smem > 0) {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<T, CPL, true>, 512,
                                                      smem);
    if (e != cudaSuccess) return e;
    per_sm = per_sm < 1 ? 1 : per_sm;
    score_kernel<T, CPL, true><<<a.num_sms * per_sm, 512, smem, st>>>(a);
  } else {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<T, CPL, false>, 512,
                                                      0);
    if (e != cudaSuccess) return e;
    per_sm = per_sm < 1 ? 1 : per_sm;
    score_kernel<T, CPL, false><<<a.num_sms * per_sm, 512, 0, st>>>(a);
  }
  return cudaGetLastError();
}

template <typename T, int CPL>
cudaError_t dispatch_mean(const ScoreArgs& a, cudaStream_t st) {
  const int64_t threads = a.n_slabs * a.p * 16;
  recent_mean_kernel<T, CPL><<<static_cast<unsigned>((threads + 255) / 256), 256, 0, st>>>(a);
  return cudaGetLastError();
}

int chunks_per_lane(int D, int is_bf16) {
  const int n_chunks = D * (is_bf16 ? 2 : 4) / 16;
  return n_chunks <= 16 ? 1 : n_chunks <= 32 ? 2 : n_chunks <= 64 ? 4 : 8;
}

template <typename T>
cudaError_t prepare_t() {
  const int bytes = static_cast<int>(kScoreSmemLimit);
  cudaError_t e;
  if ((e = cudaFuncSetAttribute(score_kernel<T, 1, true>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(score_kernel<T, 2, true>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  if ((e = cudaFuncSetAttribute(score_kernel<T, 4, true>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize, bytes)) != cudaSuccess)
    return e;
  return cudaFuncSetAttribute(score_kernel<T, 8, true>,
                              cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
}

}  // namespace

size_t score_smem_bytes(int p, int D) {
  const size_t b = static_cast<size_t>(p) * D * sizeof(float);
  return b <= kScoreSmemLimit ? b : 0;  // 0: m is read through L2 instead
}

cudaError_t score_prepare(int, int) {
  cudaError_t e = prepare_t<uint16_t>();
  return e != cudaSuccess ? e : prepare_t<float>();
}

cudaError_t launch_recent_mean(const ScoreArgs& a, cudaStream_t st) {
  const int cpl = chunks_per_lane(a.D, a.is_bf16);
  if (a.is_bf16) {
    switch (cpl) {
      case 1: return dispatch_mean<uint16_t, 1>(a, st);
      case 2: return dispatch_mean<uint16_t, 2>(a, st);
      case 4: return dispatch_mean<uint16_t, 4>(a, st);
      default: return dispatch_mean<uint16_t, 8>(a, st);
    }
  }
  switch (cpl) {
    case 1: return dispatch_mean<float, 1>(a, st);
    case 2: return dispatch_mean<float, 2>(a, st);
    case 4: return dispatch_mean<float, 4>(a, st);
    default: return dispatch_mean<float, 8>(a, st);
  }
}

cudaError_t launch_score(const ScoreArgs& a, cudaStream_t st) {
  const int cpl = chunks_per_lane(a.D, a.is_bf16);
  if (a.is_bf16) {
    switch (cpl) {
      case 1: return dispatch_score<uint16_t, 1>(a, st);
      case 2: return dispatch_score<uint16_t, 2>(a, st);
      case 4: return dispatch_score<uint16_t, 4>(a, st);
      default: return dispatch_score<uint16_t, 8>(a, st);
    }
  }
  switch (cpl) {
    case 1: return dispatch_score<float, 1>(a, st);
    case 2: return dispatch_score<float, 2>(a, st);
    case 4: return dispatch_score<float, 4>(a, st);
    default: return dispatch_score<float, 8>(a, st);
  }
}

}  // namespace ipv
