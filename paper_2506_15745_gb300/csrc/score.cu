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
#include "ipv_common.cuh"

namespace ipv {
namespace {

// Row layout: a K or V row is n_chunks 16-byte chunks. LPR lanes share a row;
// lane `sub` of the group owns chunks sub, sub + LPR, ... (CPL of them), so
// each load instruction of the group reads LPR*16 contiguous bytes. A warp
// covers 32/LPR rows per step.
template <int LPR>
__device__ __forceinline__ float group_sum(float x) {
#pragma unroll
  for (int off = 1; off < LPR; off <<= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  return x;
}

// m_q = (1/r) sum_t' k_t' / max(|k_t'|, eps) over the r recent rows
// n_past + t' p + q of each (slab, patch q). A warp handles 32/LPR patches,
// one per lane group; each group walks its r rows kBatch at a time.
template <typename T, int LPR, int CPL>
__global__ void __launch_bounds__(128) recent_mean_kernel(ScoreArgs a) {
  constexpr int P2 = Chunk<T>::kPairs;
  constexpr int E = Chunk<T>::kElems;
  constexpr int RPW = 32 / LPR;
  constexpr int kBatch = 3;
  const int lane = threadIdx.x & 31;
  const int sub = lane % LPR, grp = lane / LPR;
  const int64_t warp = (blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x) >> 5;
  const int64_t col = warp * RPW + grp;
  const bool col_ok = col < a.n_slabs * a.p;
  const int64_t s = col_ok ? col / a.p : 0;
  const int q = col_ok ? static_cast<int>(col - s * a.p) : 0;
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int64_t n_past = a.n_tokens - static_cast<int64_t>(a.r) * a.p;
  const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;

  float2 acc[CPL][P2];
#pragma unroll
  for (int i = 0; i < CPL; ++i)
#pragma unroll
    for (int e = 0; e < P2; ++e) acc[i][e] = make_float2(0.0f, 0.0f);

  for (int t0 = 0; t0 < a.r; t0 += kBatch) {  // uniform across the warp
    uint4 raw[kBatch][CPL];
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      const bool ok = col_ok && t0 + b < a.r;
      const char* row = kslab + (n_past + static_cast<int64_t>(t0 + b) * a.p + q) * row_bytes;
#pragma unroll
      for (int i = 0; i < CPL; ++i) {
        const int c = sub + LPR * i;
        raw[b][i] = (ok && c < n_chunks) ? ld_stream(row + c * 16) : make_uint4(0, 0, 0, 0);
      }
    }
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      float2 x[CPL][P2];
      float2 kk2 = make_float2(0.0f, 0.0f);
#pragma unroll
      for (int i = 0; i < CPL; ++i) {
        Chunk<T>::widen2(raw[b][i], x[i]);
#pragma unroll
        for (int e = 0; e < P2; ++e) kk2 = fma2(x[i][e], x[i][e], kk2);
      }
      const float kk = group_sum<LPR>(kk2.x + kk2.y);
      // 1 / max(|k|, eps) = rsqrt(max(|k|^2, eps^2)); rows past r contribute 0.
      const float inv = (t0 + b < a.r) ? rsqrtf(fmaxf(kk, kNormEps * kNormEps)) : 0.0f;
      const float2 inv2 = make_float2(inv, inv);
#pragma unroll
      for (int i = 0; i < CPL; ++i)
#pragma unroll
        for (int e = 0; e < P2; ++e) acc[i][e] = fma2(x[i][e], inv2, acc[i][e]);
    }
  }
  if (!col_ok) return;
  const float inv_r = 1.0f / static_cast<float>(a.r);
  float* mrow = a.m + (s * a.p + q) * static_cast<int64_t>(a.D);
#pragma unroll
  for (int i = 0; i < CPL; ++i) {
    const int c = sub + LPR * i;
    if (c < n_chunks) {
#pragma unroll
      for (int e = 0; e < P2; e += 2)
        *reinterpret_cast<float4*>(mrow + c * E + 2 * e) =
            make_float4(acc[i][e].x * inv_r, acc[i][e].y * inv_r, acc[i][e + 1].x * inv_r,
                        acc[i][e + 1].y * inv_r);
    }
  }
  if (a.zero_recent && sub == 0) {
    for (int t = 0; t < a.r; ++t) {
      const int64_t n = n_past + static_cast<int64_t>(t) * a.p + q;
      a.tar[s * a.n_tokens + n] = 0.0f;
      a.van[s * a.n_tokens + n] = 0.0f;
    }
  }
}

// Streams the past rows. Block b owns an equal contiguous share of the
// flattened (slab, past row) space; for each slab its share touches, the
// slab's m table is staged in shared memory with rows padded to D+4 floats
// (SMEM_M), or read through L1/L2. Each warp step covers 32/LPR consecutive
// rows; kU steps are loaded before any is reduced.
template <typename T, int LPR, int CPL, bool SMEM_M>
__global__ void __launch_bounds__(512, 1) score_kernel(ScoreArgs a) {
  constexpr int E = Chunk<T>::kElems;
  constexpr int P2 = Chunk<T>::kPairs;
  constexpr int RPW = 32 / LPR;
  constexpr int kU = CPL >= 8 ? 1 : 8 / CPL;
  extern __shared__ float4 sm_m4[];
  const int lane = threadIdx.x & 31;
  const int sub = lane % LPR, grp = lane / LPR;
  const int warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int ms = SMEM_M ? a.D + 4 : a.D;  // m row stride (floats)
  const int p = a.p;
  const int64_t n_past = a.n_tokens - static_cast<int64_t>(a.r) * p;
  const int64_t total = a.n_slabs * n_past;
  const int64_t end = total * (blockIdx.x + 1) / gridDim.x;
  int64_t pos = total * blockIdx.x / gridDim.x;
  const int step = n_warps * RPW * kU;  // rows per block iteration
  // Row offsets of this lane within a block iteration, and their residues mod p.
  int off[kU], off_mod[kU];
#pragma unroll
  for (int u = 0; u < kU; ++u) {
    off[u] = (u * n_warps + warp) * RPW + grp;
    off_mod[u] = off[u] % p;
  }
  const int step_mod = step % p;

  while (pos < end) {  // block-uniform
    const int64_t s = pos / n_past;
    const int lo = static_cast<int>(pos - s * n_past);
    const int hi = static_cast<int>(min(n_past, static_cast<int64_t>(lo) + (end - pos)));
    const float* m_slab = a.m + s * p * static_cast<int64_t>(a.D);
    if (SMEM_M) {
      __syncthreads();  // the previous slab's table is no longer read
      const int d4 = a.D / 4;
      for (int q = warp; q < p; q += n_warps) {
        const float4* src = reinterpret_cast<const float4*>(m_slab + static_cast<int64_t>(q) * a.D);
        float4* dst = sm_m4 + q * (ms / 4);
        for (int j = lane; j < d4; j += 32) dst[j] = __ldg(src + j);
      }
      __syncthreads();
    }
    const float* mtab = SMEM_M ? reinterpret_cast<const float*>(sm_m4) : m_slab;
    const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;
    const char* vslab = static_cast<const char*>(a.v) + s * a.cap * row_bytes;
    const uint16_t* pid = a.patch_id ? a.patch_id + s * a.cap : nullptr;
    float* tar = a.tar + s * a.n_tokens;
    float* van = a.van + s * a.n_tokens;
    int q_base = lo % p;

    for (int base = lo; base < hi; base += step) {  // block-uniform trip count
      uint4 kr[kU][CPL], vr[kU][CPL];
      int q[kU];
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int n = base + off[u];
        const bool ok = n < hi;
        const int64_t ro = static_cast<int64_t>(n) * row_bytes;
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
          const int c = sub + LPR * i;
          const bool ld = ok && c < n_chunks;
          kr[u][i] = ld ? ld_stream(kslab + ro + c * 16) : make_uint4(0, 0, 0, 0);
          vr[u][i] = ld ? ld_stream(vslab + ro + c * 16) : make_uint4(0, 0, 0, 0);
        }
        int qi = q_base + off_mod[u];
        qi = qi >= p ? qi - p : qi;
        q[u] = pid ? (ok ? static_cast<int>(pid[n]) : 0) : qi;
      }
#pragma unroll
      for (int u = 0; u < kU; ++u) {
        const int n = base + off[u];
        const bool q_ok = q[u] < p;
        const float* mq = mtab + (q_ok ? q[u] : 0) * ms;
        float2 dot2 = make_float2(0.0f, 0.0f), kk2 = dot2, vv2 = dot2;
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
          const int c = sub + LPR * i;
          float2 kx[P2], vx[P2];
          Chunk<T>::widen2(kr[u][i], kx);
          Chunk<T>::widen2(vr[u][i], vx);
          if (c < n_chunks) {
#pragma unroll
            for (int e = 0; e < P2; e += 2) {
              const float4 mv = SMEM_M ? *reinterpret_cast<const float4*>(mq + c * E + 2 * e)
                                       : __ldg(reinterpret_cast<const float4*>(mq + c * E + 2 * e));
              dot2 = fma2(kx[e], make_float2(mv.x, mv.y), dot2);
              dot2 = fma2(kx[e + 1], make_float2(mv.z, mv.w), dot2);
            }
          }
#pragma unroll
          for (int e = 0; e < P2; ++e) {
            kk2 = fma2(kx[e], kx[e], kk2);
            vv2 = fma2(vx[e], vx[e], vv2);
          }
        }
        const float dot = group_sum<LPR>(dot2.x + dot2.y);
        const float kk = group_sum<LPR>(kk2.x + kk2.y);
        const float vv = group_sum<LPR>(vv2.x + vv2.y);
        if (sub == 0 && n < hi) {
          // max(|k|, eps) = sqrt(max(|k|^2, eps^2)). A patch id outside
          // [0, p) has no recent-frame partner: NaN scores rank below every
          // number, so such a token is never preferred.
          tar[n] = q_ok ? -dot * rsqrtf(fmaxf(kk, kNormEps * kNormEps)) : __int_as_float(0x7fc00000);
          van[n] = q_ok ? sqrtf(vv) : __int_as_float(0x7fc00000);
        }
      }
      q_base += step_mod;
      q_base = q_base >= p ? q_base - p : q_base;
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
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<T, LPR, CPL, true>, 512,
                                                      smem);
    if (e != cudaSuccess) return e;
    per_sm = per_sm < 1 ? 1 : per_sm;
    score_kernel<T, LPR, CPL, true><<<a.num_sms * per_sm, 512, smem, st>>>(a);
  } else {
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, score_kernel<T, LPR, CPL, false>,
                                                      512, 0);
    if (e != cudaSuccess) return e;
    per_sm = per_sm < 1 ? 1 : per_sm;
    score_kernel<T, LPR, CPL, false><<<a.num_sms * per_sm, 512, 0, st>>>(a);
  }
  return cudaGetLastError();
}

template <typename T, int LPR, int CPL>
cudaError_t dispatch_mean(const ScoreArgs& a, cudaStream_t st) {
  const int64_t warps = (a.n_slabs * a.p + (32 / LPR) - 1) / (32 / LPR);
  recent_mean_kernel<T, LPR, CPL><<<static_cast<unsigned>((warps * 32 + 127) / 128), 128, 0, st>>>(a);
  return cudaGetLastError();
}

// (lanes per row, chunks per lane) for a row of n_chunks 16-byte chunks.
int row_shape(int D, int is_bf16) {
  const int n_chunks = D * (is_bf16 ? 2 : 4) / 16;
  return n_chunks <= 4 ? 41 : n_chunks <= 8 ? 42 : n_chunks <= 16 ? 44 : n_chunks <= 32 ? 84
         : n_chunks <= 64 ? 164 : 168;
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
  switch (row_shape(a.D, a.is_bf16)) {
    case 41: return MEAN ? dispatch_mean<T, 4, 1>(a, st) : dispatch_score<T, 4, 1>(a, st);
    case 42: return MEAN ? dispatch_mean<T, 4, 2>(a, st) : dispatch_score<T, 4, 2>(a, st);
    case 44: return MEAN ? dispatch_mean<T, 4, 4>(a, st) : dispatch_score<T, 4, 4>(a, st);
    case 84: return MEAN ? dispatch_mean<T, 8, 4>(a, st) : dispatch_score<T, 8, 4>(a, st);
    case 164: return MEAN ? dispatch_mean<T, 16, 4>(a, st) : dispatch_score<T, 16, 4>(a, st);
    default: return MEAN ? dispatch_mean<T, 16, 8>(a, st) : dispatch_score<T, 16, 8>(a, st);
  }
}

}  // namespace

size_t score_smem_bytes(int p, int D) {
  const size_t b = static_cast<size_t>(p) * (D + 4) * sizeof(float);
  return b <= kScoreSmemLimit ? b : 0;  // 0: m is read through L1/L2 instead
}

cudaError_t score_prepare(int, int) {
  cudaError_t e = prepare_t<uint16_t>();
  return e != cudaSuccess ? e : prepare_t<float>();
}

cudaError_t launch_recent_mean(const ScoreArgs& a, cudaStream_t st) {
  return a.is_bf16 ? dispatch_t<uint16_t, true>(a, st) : dispatch_t<float, true>(a, st);
}

cudaError_t launch_score(const ScoreArgs& a, cudaStream_t st) {
  return a.is_bf16 ? dispatch_t<uint16_t, false>(a, st) : dispatch_t<float, false>(a, st);
}

}  // namespace ipv
