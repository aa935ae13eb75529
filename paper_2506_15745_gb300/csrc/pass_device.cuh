// Device building blocks of the compression pass, shared by the step kernels
// (score.cu, select.cu, gather.cu) and the fused pass (window.cu), so that
// both paths run exactly the same arithmetic.
#pragma once

#include "ipv_common.cuh"

namespace ipv {
namespace dev {

// ------------------------------------------------------------------ scoring
// Row layout: a K or V row is n_chunks 16-byte chunks. LPR lanes share a row;
// lane `sub` of the group owns chunks sub, sub + LPR, ... (CPL of them), so
// each load instruction of the group reads LPR*16 contiguous bytes.
template <int LPR>
__device__ __forceinline__ float group_sum(float x) {
#pragma unroll
  for (int off = 1; off < LPR; off <<= 1) x += __shfl_xor_sync(0xffffffffu, x, off);
  return x;
}

// Recent-frame mean of one patch per lane group (warp-level: every lane of
// the warp calls it). Sec. 3.1 Eq. (tar) regrouped:
//   m_q = (1/r) sum_t' k_t' / max(|k_t'|, eps),  rows n_past + t' p + q.
// col_ok false: the group has no column (it still joins the shuffles).
// VIRT (the shared index set): s is a layer of a.hs heads and a token's key
// is its hs head-rows read as one vector (Sec. 3.1, K in R^{H x N x D}): chunk
// c of the group is chunk c mod cph of head c / cph, the norm runs over all
// heads, and each head's part of m_q goes to that head-slab's table.
template <typename T, int LPR, int CPL, bool VIRT = false>
__device__ __forceinline__ void mean_group(const ScoreArgs& a, int64_t s, int q, bool col_ok) {
  constexpr int P2 = Chunk<T>::kPairs;
  constexpr int E = Chunk<T>::kElems;
  constexpr int kBatch = 3;
  const int lane = threadIdx.x & 31;
  const int sub = lane % LPR;
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int cph = row_bytes / 16;                 // chunks of one head-row
  const int hs = VIRT ? a.hs : 1;
  const int n_chunks = cph * hs;
  const int64_t n_past = a.n_tokens - static_cast<int64_t>(a.r) * a.p;
  const int64_t slab0 = s * hs;                   // first head-slab of this token block
  const char* kslab = static_cast<const char*>(a.k) + slab0 * a.cap * row_bytes;
  int64_t coff[CPL];  // VIRT: byte offset of each chunk in a token block (else c * 16, inline)
  if (VIRT) {
#pragma unroll
    for (int i = 0; i < CPL; ++i) {
      const int c = sub + LPR * i;
      const int h = c / cph;
      coff[i] = static_cast<int64_t>(h) * a.cap * row_bytes + (c - h * cph) * 16;
    }
  }

  float2 acc[CPL][P2];
#pragma unroll
  for (int i = 0; i < CPL; ++i)
#pragma unroll
    for (int e = 0; e < P2; ++e) acc[i][e] = make_float2(0.0f, 0.0f);

  // The recent K rows stay in L2 (evict-last) for the compaction, which
  // copies them later in the pass; the scan in between is evict-first.
  const uint64_t keep = l2_evict_last();
  for (int t0 = 0; t0 < a.r; t0 += kBatch) {  // uniform across the warp
    uint4 raw[kBatch][CPL];
#pragma unroll
    for (int b = 0; b < kBatch; ++b) {
      const bool ok = col_ok && t0 + b < a.r;
      const char* row = kslab + (n_past + static_cast<int64_t>(t0 + b) * a.p + q) * row_bytes;
#pragma unroll
      for (int i = 0; i < CPL; ++i) {
        const int c = sub + LPR * i;
        raw[b][i] = (ok && c < n_chunks) ? ld_stream(row + (VIRT ? coff[i] : c * 16), keep)
                                         : make_uint4(0, 0, 0, 0);
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
  if (a.van_recent) {  // VaN of the r recent rows of patch q (Sec. 3.2), for a layer's CV
    const char* vslab = static_cast<const char*>(a.v) + slab0 * a.cap * row_bytes;
    for (int t0 = 0; t0 < a.r; t0 += kBatch) {  // uniform across the warp
      uint4 raw[kBatch][CPL];
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        const bool ok = col_ok && t0 + b < a.r;
        const char* row = vslab + (n_past + static_cast<int64_t>(t0 + b) * a.p + q) * row_bytes;
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
          const int c = sub + LPR * i;
          raw[b][i] = (ok && c < n_chunks) ? ld_stream(row + (VIRT ? coff[i] : c * 16)) : make_uint4(0, 0, 0, 0);
        }
      }
#pragma unroll
      for (int b = 0; b < kBatch; ++b) {
        float2 vv2 = make_float2(0.0f, 0.0f);
#pragma unroll
        for (int i = 0; i < CPL; ++i) {
          float2 x[P2];
          Chunk<T>::widen2(raw[b][i], x);
#pragma unroll
          for (int e = 0; e < P2; ++e) vv2 = fma2(x[e], x[e], vv2);
        }
        const float vv = group_sum<LPR>(vv2.x + vv2.y);
        if (col_ok && sub == 0 && t0 + b < a.r)
          a.van[s * a.n_tokens + n_past + static_cast<int64_t>(t0 + b) * a.p + q] = sqrtf(vv);
      }
    }
  }
  if (!col_ok) return;
  const float inv_r = 1.0f / static_cast<float>(a.r);
#pragma unroll
  for (int i = 0; i < CPL; ++i) {
    const int c = sub + LPR * i;
    if (c < n_chunks) {
      const int h = VIRT ? c / cph : 0;
      const int cc = c - h * cph;
      float* mrow = a.m + ((slab0 + h) * a.p + q) * static_cast<int64_t>(a.D);
#pragma unroll
      for (int e = 0; e < P2; e += 2)
        *reinterpret_cast<float4*>(mrow + cc * E + 2 * e) =
            make_float4(acc[i][e].x * inv_r, acc[i][e].y * inv_r, acc[i][e + 1].x * inv_r,
                        acc[i][e + 1].y * inv_r);
    }
  }
  if (a.zero_recent && sub == 0) {
    for (int t = 0; t < a.r; ++t) {
      const int64_t n = n_past + static_cast<int64_t>(t) * a.p + q;
      a.tar[s * a.n_tokens + n] = 0.0f;
      if (!a.van_recent) a.van[s * a.n_tokens + n] = 0.0f;
    }
  }
}

// Where score_segment reads the m table from.
enum MSource { kMSmem = 0, kMGlobalRO = 1, kMGlobal = 2 };

template <int MSRC>
__device__ __forceinline__ float4 load_m4(const float* p) {
  if (MSRC == kMSmem) return *reinterpret_cast<const float4*>(p);
  if (MSRC == kMGlobalRO) return __ldg(reinterpret_cast<const float4*>(p));
  return *reinterpret_cast<const float4*>(p);  // written earlier in the same kernel
}

// The three sums of one row, reduced over its LPR lanes: k.m_q, |k|^2 and
// |v|^2 (fp32, packed FMA per lane in chunk order, then a shuffle tree). kr
// and vr hold the lane's CPL chunks of the K and V row; mq is the row's m_q.
// Every scoring path uses this function, so all give the same bits.
template <typename T, int LPR, int CPL, int MSRC>
__device__ __forceinline__ void row_sums(const uint4* kr, const uint4* vr, const float* mq, int sub,
                                         int n_chunks, float* dot, float* kk, float* vv) {
  constexpr int E = Chunk<T>::kElems;
  constexpr int P2 = Chunk<T>::kPairs;
  float2 dot2 = make_float2(0.0f, 0.0f), kk2 = dot2, vv2 = dot2;
#pragma unroll
  for (int i = 0; i < CPL; ++i) {
    const int c = sub + LPR * i;
    float2 kx[P2], vx[P2];
    Chunk<T>::widen2(kr[i], kx);
    Chunk<T>::widen2(vr[i], vx);
    if (c < n_chunks) {
#pragma unroll
      for (int e = 0; e < P2; e += 2) {
        const float4 mv = load_m4<MSRC>(mq + c * E + 2 * e);
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
  *dot = group_sum<LPR>(dot2.x + dot2.y);
  *kk = group_sum<LPR>(kk2.x + kk2.y);
  *vv = group_sum<LPR>(vv2.x + vv2.y);
}

// Sec. 3.1 Eq. (tar) and Sec. 3.2 from a row's sums: s_TaR = -(k . m_q) /
// max(|k|, eps), with max(|k|, eps) = sqrt(max(|k|^2, eps^2)); s_VaN = |v|.
__device__ __forceinline__ float tar_of(float dot, float kk) {
  return -dot * rsqrtf(fmaxf(kk, kNormEps * kNormEps));
}

// TaR and VaN of past rows [lo, hi) of slab s by every warp of the block
// (block-uniform arguments). Sec. 3.1 Eq. (tar): s_TaR = -(k . m_q) / max(|k|, eps);
// Sec. 3.2: s_VaN = |v|. Each warp step covers 32/LPR consecutive rows; kU
// steps are loaded before any is reduced. mtab rows are ms floats apart.
template <typename T, int LPR, int CPL, int kU, int MSRC>
__device__ __forceinline__ void score_segment(const ScoreArgs& a, int64_t s, int lo, int hi,
                                              const float* mtab, int ms) {
  constexpr int RPW = 32 / LPR;
  const int lane = threadIdx.x & 31;
  const int sub = lane % LPR, grp = lane / LPR;
  const int warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int p = a.p;
  const int step = n_warps * RPW * kU;
  int off[kU], off_mod[kU];
#pragma unroll
  for (int u = 0; u < kU; ++u) {
    off[u] = (u * n_warps + warp) * RPW + grp;
    off_mod[u] = off[u] % p;
  }
  const int step_mod = step % p;
  const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;
  const char* vslab = static_cast<const char*>(a.v) + s * a.cap * row_bytes;
  const uint16_t* pid = a.patch_id ? a.patch_id + s * a.cap : nullptr;
  float* tar = a.tar + s * a.n_tokens;
  float* van = a.van + s * a.n_tokens;
  int q_base = lo % p;
  const uint64_t once = l2_evict_first();  // read once: keep L2 for the recent rows

  for (int base = lo; base < hi; base += step) {
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
        kr[u][i] = ld ? ld_stream(kslab + ro + c * 16, once) : make_uint4(0, 0, 0, 0);
        vr[u][i] = ld ? ld_stream(vslab + ro + c * 16, once) : make_uint4(0, 0, 0, 0);
      }
      int qi = q_base + off_mod[u];
      qi = qi >= p ? qi - p : qi;
      q[u] = pid ? (ok ? static_cast<int>(pid[n]) : 0) : qi;
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int n = base + off[u];
      const bool q_ok = q[u] < p;
      const float* mq = mtab + static_cast<int64_t>(q_ok ? q[u] : 0) * ms;
      float dot, kk, vv;
      row_sums<T, LPR, CPL, MSRC>(kr[u], vr[u], mq, sub, n_chunks, &dot, &kk, &vv);
      if (sub == 0 && n < hi) {
        // A patch id outside [0, p) has no recent-frame partner: NaN scores
        // rank below every number, so such a token is never preferred.
        if (a.kk) {  // the shared index set: this head's partial sums
          tar[n] = q_ok ? dot : __int_as_float(0x7fc00000);
          a.kk[s * a.n_tokens + n] = kk;
          van[n] = q_ok ? vv : __int_as_float(0x7fc00000);
        } else {
          tar[n] = q_ok ? tar_of(dot, kk) : __int_as_float(0x7fc00000);
          van[n] = q_ok ? sqrtf(vv) : __int_as_float(0x7fc00000);
        }
      }
    }
    q_base += step_mod;
    q_base = q_base >= p ? q_base - p : q_base;
  }
}

// TaR and VaN of the past rows of patches [q0, q0 + nq) of slab s, for a
// cache that has never been compacted (row n = f p + q; f < f_past) by every
// warp of the block. mtab holds m_q of those patches, row q - q0 at
// (q - q0) * ms floats (shared memory). Same arithmetic as score_segment.
template <typename T, int LPR, int CPL>
__device__ __forceinline__ void score_patch_rows(const ScoreArgs& a, int64_t s, int q0, int nq, int f_past,
                                                 const float* mtab, int ms) {
  constexpr int RPW = 32 / LPR;
  const int lane = threadIdx.x & 31;
  const int sub = lane % LPR, grp = lane / LPR;
  const int warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int n_rows = f_past * nq;
  const int G = n_warps * RPW;
  const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;
  const char* vslab = static_cast<const char*>(a.v) + s * a.cap * row_bytes;
  float* tar = a.tar + s * a.n_tokens;
  float* van = a.van + s * a.n_tokens;
  for (int base = 0; base < n_rows; base += G) {  // warp-uniform
    const int i = base + warp * RPW + grp;
    const bool ok = i < n_rows;
    const int f = ok ? i / nq : 0;
    const int qi = ok ? i - f * nq : 0;
    const int64_t n = static_cast<int64_t>(f) * a.p + q0 + qi;
    uint4 kr[CPL], vr[CPL];
#pragma unroll
    for (int c = 0; c < CPL; ++c) {
      const int ch = sub + LPR * c;
      const bool ld = ok && ch < n_chunks;
      kr[c] = ld ? ld_stream(kslab + n * row_bytes + ch * 16) : make_uint4(0, 0, 0, 0);
      vr[c] = ld ? ld_stream(vslab + n * row_bytes + ch * 16) : make_uint4(0, 0, 0, 0);
    }
    float dot, kk, vv;
    row_sums<T, LPR, CPL, kMSmem>(kr, vr, mtab + qi * ms, sub, n_chunks, &dot, &kk, &vv);
    if (sub == 0 && ok) {
      tar[n] = tar_of(dot, kk);
      van[n] = sqrtf(vv);
    }
  }
}

// ------------------------------------------------------------------ selection
// Per slab (Sec. 3.3; Algorithm 1 steps 3-5): keep the r p recent tokens,
// take the n_tar past tokens of highest s_TaR, then the n_van past tokens of
// highest s_VaN among those TaR left (Algorithm 2's max-forcing of TaR picks
// before its final TopK). Ties go to the lower index; NaN ranks lowest.
//
// One block of NT threads per slab; scores live in shared memory as
// order-preserving uint32 keys. A stage finds its k winners without a sort,
// from a 2048-bin histogram whose bins are a monotone map of the score (so
// every bin above the one holding the k-th winner is taken whole):
//   TaR, a mean of cosines in [-1, 1]: 2048 equal bins over [-1, 1], values
//        outside folded into the end bins, so that its histogram is built in
//        the pass that loads the scores;
//   VaN: 2048 equal bins over [min, max] of every past token's VaN, a range
//        taken in that same pass (the VaN stage's candidates are a subset).
// The candidates of the boundary bin are ranked exactly against each other
// with the index tie-break. A boundary bin of more than NT candidates falls
// back to an exact search over integer key windows with ties counted by a
// block-wide prefix sum in index order. Any score values are handled
// exactly; the bins only decide how much work the exact steps have.
constexpr uint32_t kTaken = 0xFFFFFFFFu;  // VaN pick (never a score key)
constexpr uint32_t kExcluded = 0u;        // TaR pick, excluded from the VaN stage
constexpr uint32_t kNanKey = 1u;          // score_key of every NaN
constexpr uint32_t kNoBin = 0xFFFFFFFFu;

struct SelShared {
  uint32_t warp_a[32];
  uint32_t warp_b[32];
  float warp_f[32];
  float warp_g[32];
  uint32_t bcast[8];
  float fcast[2];
  uint32_t list_n;
};

// Shared memory of select_slab: keys[pad4(n_past)], hist_tar[2048],
// hist_van[2048], list_key[NT], list_idx[NT], and with a.van_smem the VaN
// scores[pad4(n_past)].
template <int NT>
__host__ __device__ constexpr size_t select_smem_words(int64_t n_past, bool van_smem = false) {
  return static_cast<size_t>((n_past + 3) & ~3LL) * (van_smem ? 2 : 1) + 2 * kSelectBins + 2 * NT;
}

__device__ __forceinline__ bool is_cand(uint32_t k) { return k != kExcluded && k != kTaken; }

__device__ __forceinline__ float key_value(uint32_t k) {  // inverse of score_key, keys >= 2
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// A monotone non-decreasing map of a score (not NaN) to one of 2048 bins:
// floor((v - lo) * scale), folded into [0, 2047] (scale 0: every value in bin 0).
struct Bins {
  float lo, scale;
  __device__ __forceinline__ int of(float v) const {
    return static_cast<int>(fminf(fmaxf((v - lo) * scale, 0.0f), 2047.0f));
  }
};
__device__ __forceinline__ Bins tar_bins() { return Bins{-1.0f, 1024.0f}; }
__device__ __forceinline__ Bins range_bins(float vmin, float vmax) {
  const float range = vmax - vmin;
  const float scale = static_cast<float>(kSelectBins) / range;
  return Bins{vmin, (range > 0.0f && scale < INFINITY) ? scale : 0.0f};
}

__device__ __forceinline__ uint32_t warp_incl_scan(uint32_t v) {
  const int lane = threadIdx.x & 31;
#pragma unroll
  for (int off = 1; off < 32; off <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, v, off);
    if (lane >= off) v += y;
  }
  return v;
}

// Exclusive prefix sum over the block's threads in thread order; *total gets the sum.
template <int NT>
__device__ uint32_t block_excl_scan(uint32_t v, uint32_t* total, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t incl = warp_incl_scan(v);
  if (lane == 31) sh.warp_a[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = lane < W ? sh.warp_a[lane] : 0u;
    const uint32_t wi = warp_incl_scan(w);
    sh.warp_b[lane] = wi - w;
    if (lane == 31) sh.bcast[7] = wi;
  }
  __syncthreads();
  const uint32_t out = sh.warp_b[warp] + incl - v;
  *total = sh.bcast[7];
  __syncthreads();
  return out;
}

// Block-wide sum of v (every thread gets it).
template <int NT>
__device__ uint32_t block_sum(uint32_t v, SelShared& sh) {
  uint32_t tot;
  block_excl_scan<NT>(v, &tot, sh);
  return tot;
}

// Block-wide sum of *cnt, min of *lo and max of *hi (every thread gets them).
template <int NT>
__device__ void block_reduce3(uint32_t* cnt, float* lo, float* hi, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  uint32_t c = *cnt;
  float l = *lo, h = *hi;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    c += __shfl_xor_sync(0xffffffffu, c, off);
    l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
    h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
  }
  if (lane == 0) {
    sh.warp_a[warp] = c;
    sh.warp_f[warp] = l;
    sh.warp_g[warp] = h;
  }
  __syncthreads();
  if (warp == 0) {
    c = lane < W ? sh.warp_a[lane] : 0u;
    l = lane < W ? sh.warp_f[lane] : INFINITY;
    h = lane < W ? sh.warp_g[lane] : -INFINITY;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      c += __shfl_xor_sync(0xffffffffu, c, off);
      l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
      h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
    }
    if (lane == 0) {
      sh.bcast[5] = c;
      sh.fcast[0] = l;
      sh.fcast[1] = h;
    }
  }
  __syncthreads();
  *cnt = sh.bcast[5];
  *lo = sh.fcast[0];
  *hi = sh.fcast[1];
  __syncthreads();
}

template <int NT>
__device__ void block_minmax(uint32_t lo, uint32_t hi, uint32_t* out_lo, uint32_t* out_hi,
                             SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, off));
    hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, off));
  }
  if (lane == 0) {
    sh.warp_a[warp] = lo;
    sh.warp_b[warp] = hi;
  }
  __syncthreads();
  if (warp == 0) {
    lo = lane < W ? sh.warp_a[lane] : 0xFFFFFFFFu;
    hi = lane < W ? sh.warp_b[lane] : 0u;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      lo = min(lo, __shfl_xor_sync(0xffffffffu, lo, off));
      hi = max(hi, __shfl_xor_sync(0xffffffffu, hi, off));
    }
    if (lane == 0) {
      sh.bcast[0] = lo;
      sh.bcast[1] = hi;
    }
  }
  __syncthreads();
  *out_lo = sh.bcast[0];
  *out_hi = sh.bcast[1];
  __syncthreads();
}

// The bin holding the k-th largest candidate (bins scanned from the top;
// thread t owns the 2048/NT bins just below bin 2048 - t 2048/NT), the count
// of candidates in higher bins and the bin's own count. kNoBin if the
// histogram holds fewer than k.
// COPIES > 1: the histogram is that many copies of 2048 bins, summed here.
template <int NT, int COPIES = 1>
__device__ void boundary_bin(const uint32_t* hist, uint32_t k, SelShared& sh, uint32_t* bsel,
                             uint32_t* above, uint32_t* cnt_b) {
  constexpr int BPT = kSelectBins / NT;
  const int top = kSelectBins - 1 - BPT * static_cast<int>(threadIdx.x);
  uint32_t h[BPT], local = 0u;
#pragma unroll
  for (int j = 0; j < BPT; ++j) {
    h[j] = 0u;
#pragma unroll
    for (int c = 0; c < COPIES; ++c) h[j] += hist[c * kSelectBins + top - j];
    local += h[j];
  }
  if (threadIdx.x == 0) sh.bcast[2] = kNoBin;  // published by the scan's barriers
  uint32_t tot;
  uint32_t run = block_excl_scan<NT>(local, &tot, sh);
#pragma unroll
  for (int j = 0; j < BPT; ++j) {
    if (run < k && k <= run + h[j]) {
      sh.bcast[2] = static_cast<uint32_t>(top - j);
      sh.bcast[3] = run;
      sh.bcast[4] = h[j];
    }
    run += h[j];
  }
  __syncthreads();
  *bsel = sh.bcast[2];
  *above = sh.bcast[3];
  *cnt_b = sh.bcast[4];
  __syncthreads();
}

// Exact threshold search over integer key windows, from the window [lo, hi]
// holding cnt candidates of which the k largest are wanted (all candidates
// above hi are taken already). Winners: candidates with key > *T plus the
// *take_eq lowest-index ones with key == *T; *cnt_eq counts those equal to *T.
// hist is scratch. The window shrinks at least 2048-fold per round (4 rounds
// for 32-bit keys); the hard round limit only guards against a broken
// invariant.
template <int NT>
__device__ void window_search(const uint32_t* key, int n, uint32_t lo, uint32_t hi, uint32_t k,
                              uint32_t cnt, uint32_t* hist, SelShared& sh, uint32_t* T,
                              uint32_t* take_eq, uint32_t* cnt_eq) {
  for (int round = 0; round < 8; ++round) {
    if (lo == hi) break;
    const uint64_t W = static_cast<uint64_t>(hi - lo) + 1u;
    for (int b = threadIdx.x; b < kSelectBins; b += NT) hist[b] = 0u;
    __syncthreads();
    for (int i0 = threadIdx.x & ~31; i0 < n; i0 += NT) {  // warp-uniform
      const int i = i0 + (threadIdx.x & 31);
      const uint32_t x = i < n ? key[i] : kExcluded;
      const bool in = i < n && x >= lo && x <= hi;
      if (in) atomicAdd(&hist[(static_cast<uint64_t>(x - lo) * kSelectBins) / W], 1u);
    }
    __syncthreads();
    uint32_t bsel, above, cnt_b;
    boundary_bin<NT>(hist, k, sh, &bsel, &above, &cnt_b);
    if (bsel == kNoBin) break;  // fewer candidates than k: cannot happen
    k -= above;
    // Keys x with floor((x-lo)*2048/W) == bsel form [lo + ceil(bsel W/2048), lo + ceil((bsel+1) W/2048) - 1].
    const uint32_t lo_b = lo + static_cast<uint32_t>((bsel * W + kSelectBins - 1) / kSelectBins);
    const uint32_t hi_b =
        lo + static_cast<uint32_t>(((bsel + 1) * W + kSelectBins - 1) / kSelectBins) - 1u;
    if (cnt_b == k) {  // the whole bin is taken: threshold just below it
      *T = lo_b - 1u;
      *take_eq = 0u;
      *cnt_eq = 0u;
      return;
    }
    lo = lo_b;
    hi = hi_b;
    cnt = cnt_b;
  }
  *T = lo;
  *take_eq = k;
  *cnt_eq = cnt;
}

// How a stage's winners are recognised in the marking pass (block-uniform).
struct Plan {
  int mode;  // 0 none, 1 every candidate, 2 key threshold, 3 bin threshold (+ pre-marked)
  Bins bins;
  uint32_t T, take, cnt_eq;
  int bthr;
};

// Decides a stage taking the k best of n_cand candidates (n_nan of them NaN);
// hist holds the candidates' numbers in the stage's bins. Boundary-bin
// winners found by direct ranking are marked in place with `mark`. scratch
// (2048 words) may be overwritten.
template <int NT>
__device__ Plan plan_stage(uint32_t* key, int n, uint32_t k, uint32_t n_cand, uint32_t n_nan, Bins bins,
                           const uint32_t* hist, uint32_t* scratch, uint32_t mark, uint32_t* list_key,
                           uint32_t* list_idx, SelShared& sh) {
  Plan P{};
  P.bins = bins;
  if (k == 0u) return P;
  if (k >= n_cand) {
    P.mode = 1;
    return P;
  }
  const uint32_t n_num = n_cand - n_nan;
  P.mode = 2;
  if (k > n_num) {  // every number, then the lowest-index NaNs
    P.T = kNanKey;
    P.take = k - n_num;
    P.cnt_eq = n_nan;
    return P;
  }
  uint32_t bsel, above, cnt_b;
  boundary_bin<NT>(hist, k, sh, &bsel, &above, &cnt_b);
  uint32_t lo = 2u, hi = kTaken - 1u, k_rem = k, cnt = n_num;
  if (bsel != kNoBin) {  // always: the histogram holds n_num >= k numbers
    k_rem = k - above;
    P.mode = 3;
    if (cnt_b == k_rem) {  // the whole boundary bin is taken
      P.bthr = static_cast<int>(bsel) - 1;
      return P;
    }
    P.bthr = static_cast<int>(bsel);
    const int lane = threadIdx.x & 31;
    if (threadIdx.x == 0) sh.list_n = 0u;
    __syncthreads();
    if (cnt_b <= static_cast<uint32_t>(NT)) {
      // Collect the boundary bin's candidates (a ballot per warp, one atomic).
      for (int i0 = threadIdx.x - lane; i0 < n; i0 += NT) {  // warp-uniform
        const int i = i0 + lane;
        const uint32_t x = i < n ? key[i] : kExcluded;
        const bool in = is_cand(x) && x != kNanKey && bins.of(key_value(x)) == static_cast<int>(bsel);
        const unsigned m = __ballot_sync(0xffffffffu, in);
        if (m == 0u) continue;
        uint32_t base = 0u;
        if (lane == __ffs(m) - 1) base = atomicAdd(&sh.list_n, static_cast<uint32_t>(__popc(m)));
        base = __shfl_sync(0xffffffffu, base, __ffs(m) - 1);
        if (in) {
          const uint32_t j = base + __popc(m & ((1u << lane) - 1u));
          if (j < static_cast<uint32_t>(NT)) {
            list_key[j] = x;
            list_idx[j] = static_cast<uint32_t>(i);
          }
        }
      }
      __syncthreads();
      const uint32_t m = min(sh.list_n, static_cast<uint32_t>(NT));
      // T threads rank one candidate (T m <= NT, T <= 32, aligned within a
      // warp), each against every T-th other one, then sum over the T lanes.
      uint32_t T = 32u;
      while (T > 1u && T * m > static_cast<uint32_t>(NT)) T >>= 1;
      const uint32_t cand = threadIdx.x / T, sub = threadIdx.x % T;
      uint32_t rank = 0u, kt = 0u, it = 0u;
      if (cand < m) {
        kt = list_key[cand];
        it = list_idx[cand];
        for (uint32_t j = sub; j < m; j += T) {
          const uint32_t kj = list_key[j];
          rank += (kj > kt || (kj == kt && list_idx[j] < it)) ? 1u : 0u;
        }
      }
      for (uint32_t off = T >> 1; off > 0u; off >>= 1) rank += __shfl_xor_sync(0xffffffffu, rank, off);
      if (cand < m && sub == 0u && rank < k_rem) key[it] = mark;
      __syncthreads();
      return P;
    }
    // Too many candidates in the bin: exact search inside its key range.
    uint32_t blo = 0xFFFFFFFFu, bhi = 0u;
    for (int i = threadIdx.x; i < n; i += NT) {
      const uint32_t x = key[i];
      if (is_cand(x) && x != kNanKey && bins.of(key_value(x)) == static_cast<int>(bsel)) {
        blo = min(blo, x);
        bhi = max(bhi, x);
      }
    }
    block_minmax<NT>(blo, bhi, &lo, &hi, sh);
    cnt = cnt_b;
  }
  P.mode = 2;
  window_search<NT>(key, n, lo, hi, k_rem, cnt, scratch, sh, &P.T, &P.take, &P.cnt_eq);
  return P;
}

// Number of keys equal to T in the chunks of lower-numbered threads.
template <int NT>
__device__ uint32_t ties_before(const uint32_t* key, int c0, int c1, uint32_t T, SelShared& sh) {
  uint32_t mine = 0u;
  for (int i = c0; i < c1; ++i) mine += (key[i] == T) ? 1u : 0u;
  uint32_t tot;
  return block_excl_scan<NT>(mine, &tot, sh);
}

// Per-thread walker of a plan over the chunk [c0, c1) in index order.
struct Picker {
  Plan P;
  uint32_t mark, rank;
  bool all_ties;
  __device__ bool pick(uint32_t x) {
    if (x == mark) return true;  // ranked winner of the boundary bin
    if (!is_cand(x)) return false;
    switch (P.mode) {
      case 1: return true;
      case 2:
        if (x > P.T) return true;
        if (x == P.T) return all_ties || (rank++ < P.take);
        return false;
      case 3: return x != kNanKey && P.bins.of(key_value(x)) > P.bthr;
      default: return false;
    }
  }
};

template <int NT>
__device__ Picker make_picker(const uint32_t* key, int c0, int c1, const Plan& P, uint32_t mark,
                              SelShared& sh) {
  Picker pk{P, mark, 0u, true};
  if (P.mode == 2 && P.take > 0u && P.take < P.cnt_eq) {
    pk.all_ties = false;
    pk.rank = ties_before<NT>(key, c0, c1, P.T, sh);
  } else if (P.mode == 2 && P.take == 0u) {
    pk.all_ties = false;  // nothing equal to T is taken
  }
  return pk;
}

// The whole selection of slab s by one block of NT threads. smem holds
// select_smem_words<NT>(n_past, a.van_smem) words. Scores are read through L2
// only (they may have been written earlier in the same kernel).
template <int NT>
__device__ void select_slab(const SelectArgs& a, int64_t s, uint32_t* smem, SelShared& sh) {
  constexpr int kB = 8;  // score loads in flight per thread
  const int n_past = static_cast<int>(a.n_tokens - a.rp);
  const int npad = (n_past + 3) & ~3;
  uint32_t* key = smem;
  uint32_t* hist_t = smem + npad;
  uint32_t* hist_v = hist_t + kSelectBins;
  uint32_t* list_key = hist_v + kSelectBins;
  uint32_t* list_idx = list_key + NT;
  // VaN goes to shared memory in the same pass as TaR when there is room,
  // so that the VaN stage does not wait for a second round of loads.
  float* vbuf = a.van_smem ? reinterpret_cast<float*>(list_idx + NT) : nullptr;
  const float* tar = a.tar + s * a.n_tokens;
  const float* van = a.van + s * a.n_tokens;
  const int chunk = (n_past + NT - 1) / NT;
  const int c0 = min(n_past, static_cast<int>(threadIdx.x) * chunk);
  const int c1 = min(n_past, c0 + chunk);

  for (int b = threadIdx.x; b < 2 * kSelectBins; b += NT) hist_t[b] = 0u;  // both histograms
  __syncthreads();

  // TaR keys and their histogram, and the range of VaN; kB loads of each
  // kind in flight.
  uint32_t nan_t = 0u;
  float vmin = INFINITY, vmax = -INFINITY;
  const Bins bt = tar_bins();
  for (int i0 = threadIdx.x; i0 < n_past; i0 += kB * NT) {
    float tv[kB], vv[kB];
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      const int i = i0 + b * NT;
      tv[b] = i < n_past ? __ldcg(tar + i) : 0.0f;
      vv[b] = i < n_past ? __ldcg(van + i) : 0.0f;
    }
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      const int i = i0 + b * NT;
      if (i >= n_past) break;
      const float v = (a.neg_tar ? -tv[b] : tv[b]) + 0.0f;  // NaN stays NaN, -0 becomes +0
      key[i] = score_key(v);
      if (vbuf) vbuf[i] = vv[b];
      if (v == v) {
        atomicAdd(&hist_t[bt.of(v)], 1u);
      } else {
        ++nan_t;
      }
      const float u = (a.neg_van ? -vv[b] : vv[b]) + 0.0f;
      if (u == u) {
        vmin = fminf(vmin, u);
        vmax = fmaxf(vmax, u);
      }
    }
  }
  // Its barriers also publish the keys and the histogram.
  block_reduce3<NT>(&nan_t, &vmin, &vmax, sh);
  const Bins bv = range_bins(vmin, vmax);

  // TaR stage over all past tokens.
  Plan P = plan_stage<NT>(key, n_past, static_cast<uint32_t>(a.n_tar), static_cast<uint32_t>(n_past),
                          nan_t, bt, hist_t, hist_t, kExcluded, list_key, list_idx, sh);
  Picker pk = make_picker<NT>(key, c0, c1, P, kExcluded, sh);
  // Mark TaR picks; the other past tokens take their VaN key, binned.
  uint32_t nan_v = 0u;
  for (int i0 = c0; i0 < c1; i0 += kB) {
    float vb[kB];  // issue the VaN loads of kB tokens before using any
#pragma unroll
    for (int b = 0; b < kB; ++b) vb[b] = (i0 + b < c1) ? (vbuf ? vbuf[i0 + b] : __ldcg(van + i0 + b)) : 0.0f;
#pragma unroll
    for (int b = 0; b < kB; ++b) {
      const int i = i0 + b;
      if (i >= c1) break;
      if (pk.pick(key[i])) {
        key[i] = kExcluded;
      } else {
        const float v = (a.neg_van ? -vb[b] : vb[b]) + 0.0f;
        key[i] = score_key(v);
        if (v == v) {
          atomicAdd(&hist_v[bv.of(v)], 1u);
        } else {
          ++nan_v;
        }
      }
    }
  }
  nan_v = block_sum<NT>(nan_v, sh);  // its barriers also publish the keys and the histogram

  // VaN stage over the past tokens TaR left.
  const uint32_t n_rest = static_cast<uint32_t>(n_past - a.n_tar);
  P = plan_stage<NT>(key, n_past, static_cast<uint32_t>(a.n_van), n_rest, nan_v, bv, hist_v, hist_t,
                     kTaken, list_key, list_idx, sh);
  pk = make_picker<NT>(key, c0, c1, P, kTaken, sh);
  for (int i = c0; i < c1; ++i)
    if (pk.pick(key[i])) key[i] = kTaken;
  __syncthreads();

  // Ascending kept indices: past picks, then the recent frames. Warp w
  // compacts the picks of its own contiguous index range with ballots, so
  // consecutive picks are stored by consecutive lanes.
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int span = ((n_past + W - 1) / W + 31) & ~31;  // indices per warp, a multiple of 32
  const int w0 = min(n_past, warp * span), w1 = min(n_past, w0 + span);
  uint32_t cnt = 0u;
  for (int i0 = w0; i0 < w1; i0 += 32) {  // warp-uniform
    const int i = i0 + lane;
    cnt += __popc(__ballot_sync(0xffffffffu, i < w1 && (key[i] == kExcluded || key[i] == kTaken)));
  }
  if (lane == 0) sh.warp_a[warp] = cnt;
  __syncthreads();
  if (warp == 0) {
    const uint32_t v = lane < W ? sh.warp_a[lane] : 0u;
    const uint32_t incl = warp_incl_scan(v);
    sh.warp_b[lane] = incl - v;
    if (lane == 31) sh.bcast[7] = incl;
  }
  __syncthreads();
  uint32_t pos = sh.warp_b[warp];
  const uint32_t total = sh.bcast[7];
  int32_t* kept = a.kept + s * a.budget;
  for (int i0 = w0; i0 < w1; i0 += 32) {
    const int i = i0 + lane;
    const bool pick = i < w1 && (key[i] == kExcluded || key[i] == kTaken);
    const uint32_t m = __ballot_sync(0xffffffffu, pick);
    const uint32_t at = pos + __popc(m & ((1u << lane) - 1u));
    if (pick && at < a.budget) kept[at] = i;
    pos += __popc(m);
  }
  // total == n_tar + n_van by construction; the recent rows follow. The
  // guards only keep a broken count from writing outside this slab's row.
  for (int64_t j = threadIdx.x; j < a.rp; j += NT)
    if (total + j < a.budget) kept[total + j] = static_cast<int32_t>(n_past + j);
  __syncthreads();  // the block's shared memory may be reused for the next slab
}

// ---------------------------------------------------------- selection, keys in registers
// The same selection with each thread holding its contiguous chunk of at
// most E past tokens in registers (chunk = ceil(n_past / NT)): every pass is
// register arithmetic, a token's bins are computed once, the boundary bin's
// candidates of a stage are collected while the stage's other tokens are
// classified, and the output positions come from one block scan of the
// threads' pick counts (chunks are in index order). For n_past <= NT * E.

// Histogram copies of the register selection: warp w adds into copy w mod
// kHistCopies, so that tokens of a popular bin contend on fewer shared-memory
// atomics (the copies are summed when the boundary bin is sought).
constexpr int kHistCopies = 4;

// Shared memory of select_slab_reg: hist_t[kHistCopies][2048],
// hist_v[kHistCopies][2048], list_key[NT], list_idx[NT], two winner bitmaps
// of ceil(n_past / 32) words.
template <int NT>
__host__ __device__ constexpr size_t select_reg_smem_words(int64_t n_past) {
  return 2 * kHistCopies * kSelectBins + 2 * NT + 2 * static_cast<size_t>((n_past + 31) / 32);
}

// Exclusive prefix sum of v over the block's threads in thread order, with
// the total, the min of lo and the max of hi over the block, in one pair of
// barriers.
template <int NT>
__device__ uint32_t block_scan_minmax(uint32_t v, uint32_t* total, float* lo, float* hi, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t incl = warp_incl_scan(v);
  float l = *lo, h = *hi;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
    h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
  }
  if (lane == 31) sh.warp_a[warp] = incl;
  if (lane == 0) {
    sh.warp_f[warp] = l;
    sh.warp_g[warp] = h;
  }
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = lane < W ? sh.warp_a[lane] : 0u;
    const uint32_t wi = warp_incl_scan(w);
    sh.warp_b[lane] = wi - w;
    l = lane < W ? sh.warp_f[lane] : INFINITY;
    h = lane < W ? sh.warp_g[lane] : -INFINITY;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
      h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
    }
    if (lane == 31) sh.bcast[7] = wi;
    if (lane == 0) {
      sh.fcast[0] = l;
      sh.fcast[1] = h;
    }
  }
  __syncthreads();
  const uint32_t out = sh.warp_b[warp] + incl - v;
  *total = sh.bcast[7];
  *lo = sh.fcast[0];
  *hi = sh.fcast[1];
  __syncthreads();
  return out;
}

// One stage over the register-resident tokens: picks the k best (key desc,
// index asc; NaN keys lowest) among the tokens whose bit is set in elig (bit
// e: token i0 + e). n_cand candidates in the block, n_nan of them NaN, and
// nan_before NaN candidates in lower-numbered threads. hist holds the
// candidates' numbers in bins (kHistCopies copies, built by the caller); scratch is 2048 words
// that may be overwritten, winmap a zeroed bitmap of ceil(n_past/32) words.
// Returns the picks as a bit mask. Block-uniform arguments except key, elig,
// nan_before.
template <int NT, int E>
__device__ uint32_t stage_reg(const uint32_t (&key)[E], uint32_t elig, int i0, uint32_t k, uint32_t n_cand,
                              uint32_t n_nan, uint32_t nan_before, Bins bins, const uint32_t* hist,
                              uint32_t* scratch, uint32_t* list_key, uint32_t* list_idx, uint32_t* winmap,
                              SelShared& sh) {
  if (k == 0u) return 0u;
  if (k >= n_cand) return elig;
  const uint32_t n_num = n_cand - n_nan;
  uint32_t pick = 0u;
  if (k > n_num) {  // every number, then the lowest-index NaNs
    const uint32_t take = k - n_num;
    uint32_t r = nan_before;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (!((elig >> e) & 1u)) continue;
      if (key[e] != kNanKey) {
        pick |= 1u << e;
      } else {
        if (r < take) pick |= 1u << e;
        ++r;
      }
    }
    return pick;
  }
  uint32_t bsel, above, cnt_b;
  boundary_bin<NT, kHistCopies>(hist, k, sh, &bsel, &above, &cnt_b);
  uint32_t k_rem = k - above;
  if (bsel != kNoBin && cnt_b == k_rem) {  // the whole boundary bin is taken
#pragma unroll
    for (int e = 0; e < E; ++e)
      if (((elig >> e) & 1u) && key[e] != kNanKey && bins.of(key_value(key[e])) >= static_cast<int>(bsel))
        pick |= 1u << e;
    return pick;
  }
  if (bsel != kNoBin && cnt_b <= static_cast<uint32_t>(NT)) {
    if (threadIdx.x == 0) sh.list_n = 0u;
    __syncthreads();
    uint32_t in_bin = 0u;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (!((elig >> e) & 1u) || key[e] == kNanKey) continue;
      const int b = bins.of(key_value(key[e]));
      if (b > static_cast<int>(bsel)) {
        pick |= 1u << e;
      } else if (b == static_cast<int>(bsel)) {
        in_bin |= 1u << e;
        const uint32_t j = atomicAdd(&sh.list_n, 1u);
        if (j < static_cast<uint32_t>(NT)) {
          list_key[j] = key[e];
          list_idx[j] = static_cast<uint32_t>(i0 + e);
        }
      }
    }
    __syncthreads();
    const uint32_t m = min(sh.list_n, static_cast<uint32_t>(NT));
    // T threads rank one candidate (T m <= NT, T <= 32, aligned within a
    // warp), each against every T-th other one, then sum over the T lanes.
    uint32_t T = 32u;
    while (T > 1u && T * m > static_cast<uint32_t>(NT)) T >>= 1;
    const uint32_t cand = threadIdx.x / T, sub = threadIdx.x % T;
    uint32_t rank = 0u, kt = 0u, it = 0u;
    if (cand < m) {
      kt = list_key[cand];
      it = list_idx[cand];
      for (uint32_t j = sub; j < m; j += T) {
        const uint32_t kj = list_key[j];
        rank += (kj > kt || (kj == kt && list_idx[j] < it)) ? 1u : 0u;
      }
    }
    for (uint32_t off = T >> 1; off > 0u; off >>= 1) rank += __shfl_xor_sync(0xffffffffu, rank, off);
    if (cand < m && sub == 0u && rank < k_rem) atomicOr(&winmap[it >> 5], 1u << (it & 31));
    __syncthreads();
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (!((in_bin >> e) & 1u)) continue;
      const int i = i0 + e;
      if ((winmap[i >> 5] >> (i & 31)) & 1u) pick |= 1u << e;
    }
    return pick;
  }
  // Boundary bin too crowded: exact search over integer key windows.
  uint32_t lo = 2u, hi = kTaken - 1u, cnt = n_num;
  if (bsel != kNoBin) {
    uint32_t blo = 0xFFFFFFFFu, bhi = 0u;
#pragma unroll
    for (int e = 0; e < E; ++e) {
      if (!((elig >> e) & 1u) || key[e] == kNanKey) continue;
      if (bins.of(key_value(key[e])) == static_cast<int>(bsel)) {
        blo = min(blo, key[e]);
        bhi = max(bhi, key[e]);
      }
    }
    block_minmax<NT>(blo, bhi, &lo, &hi, sh);
    cnt = cnt_b;
  } else {
    k_rem = k;
  }
  for (int round = 0; round < 8; ++round) {
    if (lo == hi) break;
    const uint64_t W = static_cast<uint64_t>(hi - lo) + 1u;
    for (int b = threadIdx.x; b < kSelectBins; b += NT) scratch[b] = 0u;
    __syncthreads();
#pragma unroll
    for (int e = 0; e < E; ++e) {
      const uint32_t x = key[e];
      if (((elig >> e) & 1u) && x >= lo && x <= hi)
        atomicAdd(&scratch[(static_cast<uint64_t>(x - lo) * kSelectBins) / W], 1u);
    }
    __syncthreads();
    uint32_t b2, above2, cnt2;
    boundary_bin<NT>(scratch, k_rem, sh, &b2, &above2, &cnt2);
    if (b2 == kNoBin) break;  // fewer candidates than k_rem: cannot happen
    k_rem -= above2;
    const uint32_t lo_b = lo + static_cast<uint32_t>((b2 * W + kSelectBins - 1) / kSelectBins);
    const uint32_t hi_b = lo + static_cast<uint32_t>(((b2 + 1) * W + kSelectBins - 1) / kSelectBins) - 1u;
    if (cnt2 == k_rem) {  // the whole window bin is taken: winners are keys >= lo_b
      lo = hi = lo_b - 1u;
      cnt = 0u;
      k_rem = 0u;
      break;
    }
    lo = lo_b;
    hi = hi_b;
    cnt = cnt2;
  }
  // Winners: keys above lo, and the k_rem lowest-index keys equal to lo
  // (cnt of them; all when k_rem == cnt).
  uint32_t eq = 0u;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (!((elig >> e) & 1u)) continue;
    if (key[e] > lo) pick |= 1u << e;
    if (key[e] == lo) eq |= 1u << e;
  }
  uint32_t tot;
  uint32_t r = block_excl_scan<NT>(__popc(eq), &tot, sh);
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (!((eq >> e) & 1u)) continue;
    if (r < k_rem) pick |= 1u << e;
    ++r;
  }
  return pick;
}

template <int NT, int E>
__device__ void select_slab_reg(const SelectArgs& a, int64_t s, uint32_t* smem, SelShared& sh) {
  const int n_past = static_cast<int>(a.n_tokens - a.rp);
  const int words = (n_past + 31) / 32;
  uint32_t* hist_t = smem;
  uint32_t* hist_v = hist_t + kHistCopies * kSelectBins;
  uint32_t* list_key = hist_v + kHistCopies * kSelectBins;
  uint32_t* list_idx = list_key + NT;
  uint32_t* win_t = list_idx + NT;
  uint32_t* win_v = win_t + words;
  const int copy = ((threadIdx.x >> 5) % kHistCopies) * kSelectBins;  // this warp's histogram copy
  const float* tar = a.tar + s * a.n_tokens;
  const float* van = a.van + s * a.n_tokens;
  const int chunk = (n_past + NT - 1) / NT;  // <= E
  const int i0 = min(n_past, static_cast<int>(threadIdx.x) * chunk);
  const int cnt = min(n_past - i0, chunk);
  const uint32_t mine = cnt >= 32 ? 0xFFFFFFFFu : ((1u << cnt) - 1u);

  for (int b = threadIdx.x; b < 2 * kHistCopies * kSelectBins; b += NT) hist_t[b] = 0u;  // histograms
  for (int b = threadIdx.x; b < 2 * words; b += NT) win_t[b] = 0u;                          // bitmaps
  __syncthreads();

  // Keys, TaR histogram, range of VaN. A warp's chunks are contiguous, so the
  // loads of one e across the warp share cache lines (plain loads through L1).
  // All of a thread's loads are issued before any result is used.
  uint32_t tk[E], vk[E];
#pragma unroll
  for (int e = 0; e < E; ++e) {
    tk[e] = e < cnt ? __float_as_uint(tar[i0 + e]) : 0u;
    vk[e] = e < cnt ? __float_as_uint(van[i0 + e]) : 0u;
  }
  uint32_t nan_t = 0u;
  float vmin = INFINITY, vmax = -INFINITY;
  const Bins bt = tar_bins();
#pragma unroll
  for (int e = 0; e < E; ++e) {
    const float t = __uint_as_float(tk[e]), u = __uint_as_float(vk[e]);
    const float tv = (a.neg_tar ? -t : t) + 0.0f;  // NaN stays NaN, -0 becomes +0
    const float vv = (a.neg_van ? -u : u) + 0.0f;
    tk[e] = e < cnt ? score_key(tv) : kNanKey;
    vk[e] = e < cnt ? score_key(vv) : kNanKey;
    if (e < cnt) {
      if (tv == tv) {
        atomicAdd(&hist_t[copy + bt.of(tv)], 1u);
      } else {
        ++nan_t;
      }
      if (vv == vv) {
        vmin = fminf(vmin, vv);
        vmax = fmaxf(vmax, vv);
      }
    }
  }
  uint32_t nan_t_all;
  const uint32_t nan_t_before = block_scan_minmax<NT>(nan_t, &nan_t_all, &vmin, &vmax, sh);
  const Bins bv = range_bins(vmin, vmax);

  // TaR stage over all past tokens.
  const uint32_t pick_t = stage_reg<NT, E>(tk, mine, i0, static_cast<uint32_t>(a.n_tar),
                                           static_cast<uint32_t>(n_past), nan_t_all, nan_t_before, bt, hist_t,
                                           hist_t, list_key, list_idx, win_t, sh);
  // VaN histogram of the tokens TaR left.
  const uint32_t rest = mine & ~pick_t;
  uint32_t nan_v = 0u;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (!((rest >> e) & 1u)) continue;
    if (vk[e] != kNanKey) {
      atomicAdd(&hist_v[copy + bv.of(key_value(vk[e]))], 1u);
    } else {
      ++nan_v;
    }
  }
  uint32_t nan_v_all;
  float d0 = 0.0f, d1 = 0.0f;
  const uint32_t nan_v_before = block_scan_minmax<NT>(nan_v, &nan_v_all, &d0, &d1, sh);

  // VaN stage over the past tokens TaR left.
  const uint32_t pick_v = stage_reg<NT, E>(vk, rest, i0, static_cast<uint32_t>(a.n_van),
                                           static_cast<uint32_t>(n_past - a.n_tar), nan_v_all, nan_v_before, bv,
                                           hist_v, hist_t, list_key, list_idx, win_v, sh);

  // Ascending kept indices: this thread's picks at the block prefix of the
  // counts, then the recent frames.
  const uint32_t pick = pick_t | pick_v;
  uint32_t total;
  uint32_t pos = block_excl_scan<NT>(__popc(pick), &total, sh);
  int32_t* kept = a.kept + s * a.budget;
#pragma unroll
  for (int e = 0; e < E; ++e) {
    if (!((pick >> e) & 1u)) continue;
    if (pos < a.budget) kept[pos] = i0 + e;
    ++pos;
  }
  // total == n_tar + n_van by construction; the guards only keep a broken
  // count from writing outside this slab's row.
  for (int64_t j = threadIdx.x; j < a.rp; j += NT)
    if (total + j < a.budget) kept[total + j] = static_cast<int32_t>(n_past + j);
  __syncthreads();  // the block's shared memory may be reused for the next slab
}

// ------------------------------------------------------------------ compaction
// Sec. 3.1 / Algorithm 2 last step: dst row j of a slab = src row kept[j].
// Half-warp hw (of n_hw) copies rows g = g_begin + hw, g_begin + hw + n_hw,
// ... of the flattened (slab, j) range [g_begin, g_end), kU rows in flight.
// Kept indices are read through L2 only (they may have been written earlier
// in the same kernel), source patch ids with plain loads. IDS: copy the
// patch and frame ids of each row here too (else gather_ids does it).
// JN > 0 (the step kernels): g runs over (slab, j) with j < jn kept rows per
// slab, the kept stride staying a.budget; FIXED: the source row is
// a.n_tokens - a.rp + j and kept is not read (the recent frames, j < rp,
// written to rows budget - rp + j).
template <int CPL, int kU, bool IDS = true, bool FIXED = false, bool LAST_USE = false>
__device__ __forceinline__ void gather_range(const GatherArgs& a, int64_t g_begin, int64_t g_end,
                                             int64_t hw, int64_t n_hw, int64_t jn = 0) {
  const uint64_t pol = LAST_USE ? l2_evict_first() : 0;
  const int64_t per = jn > 0 ? jn : a.budget;  // (slab, j) rows per slab in g
  const int lane = threadIdx.x & 15;
  const int n_chunks = a.row_bytes / 16;
  const char* ks = static_cast<const char*>(a.k_src);
  const char* vs = static_cast<const char*>(a.v_src);
  char* kd = static_cast<char*>(a.k_dst);
  char* vd = static_cast<char*>(a.v_dst);

  for (int64_t g0 = g_begin + hw; g0 < g_end; g0 += n_hw * kU) {
    uint4 kr[kU][CPL], vr[kU][CPL];
    int64_t dst_off[kU];
    int src_n[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int64_t g = g0 + u * n_hw;
      int n = -1;
      int64_t s = 0, j = 0;
      if (g < g_end) {
        s = g / per;
        j = g - s * per;
        if (FIXED) {
          n = static_cast<int>(a.n_tokens - a.rp + j);
          j += a.budget - a.rp;
        } else {
          n = __ldcg(a.kept + (a.heads_per_kept > 1 ? s / a.heads_per_kept : s) * a.budget + j);
        }
        if (n >= a.cap) n = -1;  // never produced by the selection; ignore
      }
      src_n[u] = n;
      dst_off[u] = (s * a.cap + j) * a.row_bytes;
      const int64_t src_off = (s * a.cap + (n < 0 ? 0 : n)) * a.row_bytes;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        const bool ld = n >= 0 && ch < n_chunks;
        if (LAST_USE) {  // the source rows are not read again in this pass
          kr[u][c] = ld ? ld_stream(ks + src_off + ch * 16, pol) : make_uint4(0, 0, 0, 0);
          vr[u][c] = ld ? ld_stream(vs + src_off + ch * 16, pol) : make_uint4(0, 0, 0, 0);
        } else {
          kr[u][c] = ld ? ld_stream(ks + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
          vr[u][c] = ld ? ld_stream(vs + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
        }
      }
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      if (src_n[u] < 0) continue;
#pragma unroll
      for (int c = 0; c < CPL; ++c) {
        const int ch = lane + 16 * c;
        if (ch < n_chunks) {
          st_stream(kd + dst_off[u] + ch * 16, kr[u][c]);
          st_stream(vd + dst_off[u] + ch * 16, vr[u][c]);
        }
      }
      if (IDS && (a.pid_dst || a.fid_dst) && lane < 2) {  // ids travel with their rows too
        const int64_t drow = dst_off[u] / a.row_bytes;       // s * cap + j
        const int64_t srow = drow - (drow % a.cap) + src_n[u];
        if (lane == 0 && a.pid_dst)
          a.pid_dst[drow] = a.pid_src ? a.pid_src[srow] : static_cast<uint16_t>(src_n[u] % a.p);
        if (lane == 1 && a.fid_dst)
          a.fid_dst[drow] = a.fid_src ? a.fid_src[srow] : static_cast<uint32_t>(src_n[u] / a.p);
      }
    }
  }
}

// Patch and frame ids of the kept rows, one (slab, j) per thread of the
// grid: consecutive j of a slab are consecutive threads, so the stores are
// coalesced (ids travel with their rows, Sec. 3.1 K~ = K[:, I, :]).
__device__ __forceinline__ void gather_ids(const GatherArgs& a) {
  if (!a.pid_dst && !a.fid_dst) return;
  const int64_t total = a.n_slabs * a.budget;
  const int64_t step = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t g = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; g < total; g += step) {
    const int64_t s = g / a.budget;
    const int64_t j = g - s * a.budget;
    const int n = a.heads_per_kept > 1 ? a.kept[(s / a.heads_per_kept) * a.budget + j] : a.kept[g];
    if (n < 0 || n >= a.cap) continue;
    const int64_t dst = s * a.cap + j;
    if (a.pid_dst)
      a.pid_dst[dst] = a.pid_src ? a.pid_src[s * a.cap + n] : static_cast<uint16_t>(n % a.p);
    if (a.fid_dst)
      a.fid_dst[dst] = a.fid_src ? a.fid_src[s * a.cap + n] : static_cast<uint32_t>(n / a.p);
  }
}

}  // namespace dev
}  // namespace ipv
