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
  uint32_t list_cnt[2];  // the register selection's list counts, one per stage
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

// 2^s as a float, for -126 <= s <= 127.
__device__ __forceinline__ float exp2_int(int s) { return __uint_as_float(static_cast<uint32_t>(s + 127) << 23); }

// A monotone non-decreasing map of a score (not NaN) to one of 2048 bins:
// floor(v mul) - off folded into [0, 2047], mul a power of two (or 0: every
// value in bin 0) and off an integer. Because v mul is exact for the values
// the bins resolve, the scores of bin b and above are those at or above
// (b + off) / mul, so a stage's boundary bin turns into two integer key
// thresholds (floor_key) and its tokens are classified by key compares.
struct Bins {
  float mul, off, inv;  // inv = 1 / mul (0 with mul)
  __device__ __forceinline__ int of(float v) const {
    return static_cast<int>(fminf(fmaxf(floorf(v * mul) - off, 0.0f), 2047.0f));
  }
  __device__ __forceinline__ bool at_least(uint32_t key, int b) const { return of(key_value(key)) >= b; }
  // The smallest number key (>= 2) whose score lies in bin b or above;
  // kTaken if there is none. The estimate from the bin's lower edge is
  // checked against its neighbour key; where rounding moved the edge, a
  // binary search over the number keys (below the key of +inf, where bin is
  // monotone) finds it. Block-uniform when b is.
  __device__ uint32_t floor_key(int b) const {
    constexpr uint32_t kInfKey = 0xFF800000u;  // score_key(+inf)
    if (b <= 0) return 2u;
    if (b >= kSelectBins || mul == 0.0f) return kTaken;
    uint32_t x = score_key((static_cast<float>(b) + off) * inv);
    x = min(max(x, 2u), kInfKey);
    if (at_least(x, b) && (x == 2u || !at_least(x - 1u, b))) return x;
    return search_key(*this, b);
  }
  __device__ static __noinline__ uint32_t search_key(Bins bins, int b) {
    constexpr uint32_t kInfKey = 0xFF800000u;
    if (!bins.at_least(kInfKey, b)) return kTaken;
    uint32_t lo = 2u, hi = kInfKey;
    while (lo < hi) {
      const uint32_t mid = lo + (hi - lo) / 2u;
      if (bins.at_least(mid, b)) {
        hi = mid;
      } else {
        lo = mid + 1u;
      }
    }
    return lo;
  }
  // The same edge as a score: bin(v) >= b exactly when v >= floor_value(b)
  // (-inf for every number, NaN, which no score reaches, for none).
  __device__ float floor_value(int b) const {
    constexpr uint32_t kNegInfKey = 0x007FFFFFu;  // score_key(-inf)
    const uint32_t x = floor_key(b);
    if (x == kTaken) return __uint_as_float(0x7FC00000u);
    return x <= kNegInfKey ? -INFINITY : key_value(x);
  }
};
// TaR (a cosine, negated) in [-1, 1]: bins of width 1/1024.
__device__ __forceinline__ Bins tar_bins() { return Bins{1024.0f, -1024.0f, 1.0f / 1024.0f}; }
// VaN over its observed range [vmin, vmax]: the largest power-of-two scale
// with (vmax - vmin) mul < 2048, kept below 2^21 |v| so that off stays an
// exact integer. One bin when there is no finite range.
__device__ __forceinline__ Bins range_bins(float vmin, float vmax) {
  const float range = vmax - vmin;
  if (!(range > 0.0f) || range == INFINITY) return Bins{0.0f, 0.0f, 0.0f};
  const auto ilog2 = [](float x) {  // floor(log2 x) for normal x > 0; -127 below
    return static_cast<int>((__float_as_uint(x) >> 23) & 0xFFu) - 127;
  };
  const int s = min(min(10 - ilog2(range), 20 - ilog2(fmaxf(fabsf(vmin), fabsf(vmax)))), 126);
  const int sc = max(s, -126);
  const float mul = exp2_int(sc);
  return Bins{mul, floorf(vmin * mul), exp2_int(-sc)};
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

// Exclusive prefix sum over the block's threads in thread order; *total gets
// the sum. Every warp scans the warp totals itself, so the scan costs two
// barriers (the second keeps warp_a from being rewritten by a next scan
// before every warp has read it).
template <int NT>
__device__ uint32_t block_excl_scan(uint32_t v, uint32_t* total, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t incl = warp_incl_scan(v);
  if (lane == 31) sh.warp_a[warp] = incl;
  __syncthreads();
  const uint32_t wt = lane < W ? sh.warp_a[lane] : 0u;
  const uint32_t wi = warp_incl_scan(wt);
  *total = __shfl_sync(0xffffffffu, wi, 31);
  const uint32_t out = __shfl_sync(0xffffffffu, wi - wt, warp) + incl - v;
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
  // Every warp reduces the warp partials itself.
  c = lane < W ? sh.warp_a[lane] : 0u;
  l = lane < W ? sh.warp_f[lane] : INFINITY;
  h = lane < W ? sh.warp_g[lane] : -INFINITY;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    c += __shfl_xor_sync(0xffffffffu, c, off);
    l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
    h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
  }
  *cnt = c;
  *lo = l;
  *hi = h;
  __syncthreads();
}

// Block-wide min of *lo and max of *hi (every thread gets them); two barriers.
template <int NT>
__device__ void block_range(float* lo, float* hi, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  float l = *lo, h = *hi;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
    h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
  }
  if (lane == 0) {
    sh.warp_f[warp] = l;
    sh.warp_g[warp] = h;
  }
  __syncthreads();
  l = lane < W ? sh.warp_f[lane] : INFINITY;
  h = lane < W ? sh.warp_g[lane] : -INFINITY;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    l = fminf(l, __shfl_xor_sync(0xffffffffu, l, off));
    h = fmaxf(h, __shfl_xor_sync(0xffffffffu, h, off));
  }
  *lo = l;
  *hi = h;
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
// thread t owns the 2048/NT bins just below bin 2048 - t 2048/NT; hist
// 16-byte aligned), the count
// of candidates in higher bins and the bin's own count. kNoBin if the
// histogram holds fewer than k.
// COPIES > 1: the histogram is that many copies of 2048 bins, summed here.
// Two barriers: bcast[2..4] and fcast are written only between them, and
// every thread reads them before it can reach the first barrier of a next
// call. With bins, the thread that finds the bin also turns its edges into
// scores (*v_lo = bins.floor_value(bin), *v_hi = that of bin + 1); *total
// gets the histogram's total.
template <int NT, int COPIES = 1>
__device__ void boundary_bin(const uint32_t* hist, uint32_t k, SelShared& sh, uint32_t* bsel,
                             uint32_t* above, uint32_t* cnt_b, const Bins* bins = nullptr,
                             float* v_lo = nullptr, float* v_hi = nullptr, uint32_t* total = nullptr) {
  constexpr int BPT = kSelectBins / NT;
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int top = kSelectBins - 1 - BPT * static_cast<int>(threadIdx.x);
  uint32_t h[BPT], local = 0u;
#pragma unroll
  for (int j = 0; j < BPT; ++j) h[j] = 0u;
  // A thread's bins are adjacent: one vector load per copy (no bank conflict
  // between lanes, which are BPT words apart).
#pragma unroll
  for (int c = 0; c < COPIES; ++c) {
    const uint32_t* hc = hist + c * kSelectBins + top - (BPT - 1);
    if constexpr (BPT == 2) {
      const uint2 x = *reinterpret_cast<const uint2*>(hc);
      h[0] += x.y;
      h[1] += x.x;
    } else if constexpr (BPT == 4) {
      const uint4 x = *reinterpret_cast<const uint4*>(hc);
      h[0] += x.w;
      h[1] += x.z;
      h[2] += x.y;
      h[3] += x.x;
    } else {
#pragma unroll
      for (int j = 0; j < BPT; ++j) h[j] += hc[BPT - 1 - j];
    }
  }
#pragma unroll
  for (int j = 0; j < BPT; ++j) local += h[j];
  const uint32_t incl = warp_incl_scan(local);
  if (lane == 31) sh.warp_a[warp] = incl;
  __syncthreads();
  const uint32_t wt = lane < W ? sh.warp_a[lane] : 0u;
  const uint32_t wi = warp_incl_scan(wt);
  const uint32_t tot = __shfl_sync(0xffffffffu, wi, 31);
  uint32_t run = __shfl_sync(0xffffffffu, wi - wt, warp) + incl - local;
  const bool finder = run < k && k <= run + local;  // the one thread holding the k-th
  int b = 0;
  if (finder) {
#pragma unroll
    for (int j = 0; j < BPT; ++j) {
      if (run < k && k <= run + h[j]) {
        b = top - j;
        sh.bcast[2] = static_cast<uint32_t>(b);
        sh.bcast[3] = run;
        sh.bcast[4] = h[j];
      }
      run += h[j];
    }
  }
  if (bins) {  // lanes 0 and 1 of the finder's warp compute the two edges side by side
    const unsigned fm = __ballot_sync(0xffffffffu, finder);
    if (fm) {
      const int bb = __shfl_sync(0xffffffffu, b, __ffs(fm) - 1);
      if (lane < 2) sh.fcast[lane] = bins->floor_value(bb + lane);
    }
  }
  __syncthreads();
  if (total) *total = tot;
  if (k == 0u || tot < k) {
    *bsel = kNoBin;
    *above = 0u;
    *cnt_b = 0u;
  } else {
    *bsel = sh.bcast[2];
    *above = sh.bcast[3];
    *cnt_b = sh.bcast[4];
    if (bins) {
      *v_lo = sh.fcast[0];
      *v_hi = sh.fcast[1];
    }
  }
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

// Largest boundary bin whose candidates are ranked against each other
// directly (m^2 / block-size comparisons per thread); a larger one, e.g. the
// whole-frame ties of frame-level scores, takes the window search over key
// bits, which is linear in the slab.
constexpr uint32_t kRankMax = 128;

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
    if (cnt_b <= kRankMax) {
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

// ---------------------------------------------------------- selection, scores in registers
// The same selection with the past tokens' scores in registers: thread t of
// NT holds tokens t, t + NT, t + 2 NT, ... (at most E; bit j of a thread's
// masks is token j NT + t, row j). Loads are coalesced; a stage's tokens
// are classified against its boundary bin by two float compares (the bin's
// edges as scores); the boundary bin's candidates are collected and ranked
// exactly; every step that needs index order (the kept order, lowest-index
// ties and NaNs) works on bitmaps whose word j W + w is warp w's ballot over
// row j, so that word order is index order. For n_past <= NT * E.

// Histogram copies of the register selection: warp w adds into copy w mod
// kHistCopies, so that tokens of a popular bin contend on fewer shared-memory
// atomics (the copies are summed when the boundary bin is sought).
constexpr int kHistCopies = 4;

// Above this many rows the VaN scores wait out the TaR stage in shared
// memory, so that the stage has the registers it needs (always, by
// default: the selection kernel runs at 48 registers).
#ifndef IPV_REG_STASH_ROWS
#define IPV_REG_STASH_ROWS 0
#endif
constexpr int kRegStashRows = IPV_REG_STASH_ROWS;

// Shared memory of select_slab_reg: hist_t[kHistCopies][2048],
// hist_v[kHistCopies][2048], list_key[NT], list_idx[NT], three bitmaps of
// E NT / 32 words (the two stages' boundary-bin winners, and a scratch one
// for index-order ranks and the picks) and, above kRegStashRows rows, the
// VaN scores (E NT words).
template <int NT, int E, bool STASH = (E > kRegStashRows)>
__host__ __device__ constexpr size_t select_reg_smem_words() {
  return 2 * kHistCopies * kSelectBins + 2 * NT + 3 * (E * NT / 32) + (STASH ? E * NT : 0);
}

// The `take` lowest-index tokens among those flagged in f (bit j: token
// j NT + t; rows j < J), as a mask. bits is scratch of J NT / 32 words.
// Block-uniform take and J.
template <int NT, int E>
__device__ __noinline__ uint32_t lowest_index(uint32_t f, uint32_t take, int J, uint32_t* bits, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const uint32_t b = __ballot_sync(0xffffffffu, (f >> j) & 1u);
    if (j < J && lane == 0) bits[j * W + warp] = b;
  }
  __syncthreads();
  // Word q's count of flagged tokens in lower words (thread q; J W <= NT).
  const uint32_t word = static_cast<int>(threadIdx.x) < J * W ? bits[threadIdx.x] : 0u;
  uint32_t tot;
  const uint32_t before = block_excl_scan<NT>(__popc(word), &tot, sh);
  if (static_cast<int>(threadIdx.x) < J * W) bits[threadIdx.x] = before;
  __syncthreads();
  const uint32_t lt = (1u << lane) - 1u;
  uint32_t out = 0u;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const uint32_t b = __ballot_sync(0xffffffffu, (f >> j) & 1u);
    if (j < J && ((f >> j) & 1u) && bits[j * W + warp] + __popc(b & lt) < take) out |= 1u << j;
  }
  __syncthreads();  // bits may be reused
  return out;
}

// One stage over the register-resident tokens: picks the k best (score desc,
// index asc; NaN lowest) among the tokens whose bit is set in elig (bit j:
// token j NT + t, score v[j], already free of -0; v is overwritten when the
// boundary bin is crowded). n_cand candidates in the block, J rows. hist
// holds the candidates' numbers in bins (kHistCopies copies, built and
// published by the caller; its total is the number of non-NaN candidates);
// scratch is 2048 words that may be overwritten, winmap a zeroed bitmap and
// bits a scratch one (J NT / 32 words each); *list_n (this stage's own
// count) is 0 on entry. Returns the picks as a bit mask. Block-uniform
// arguments except v, elig.
template <int NT, int E>
__device__ uint32_t stage_reg(float (&v)[E], uint32_t elig, int J, uint32_t k, uint32_t n_cand, Bins bins,
                              const uint32_t* hist, uint32_t* scratch, uint32_t* list_key, uint32_t* list_idx,
                              uint32_t* list_n, uint32_t* winmap, uint32_t* bits, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (k == 0u) return 0u;
  if (k >= n_cand) return elig;
  uint32_t pick = 0u;
  // The boundary bin holds the scores in [v_lo, v_hi) (NaN fails both tests).
  uint32_t bsel, above, cnt_b, n_num;
  float v_lo = 0.0f, v_hi = 0.0f;
  boundary_bin<NT, kHistCopies>(hist, k, sh, &bsel, &above, &cnt_b, &bins, &v_lo, &v_hi, &n_num);
  if (k > n_num) {  // every number, then the lowest-index NaNs
    uint32_t nan = 0u;
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const uint32_t el = (elig >> j) & 1u;
      const uint32_t num = v[j] == v[j] ? 1u : 0u;
      pick |= (el & num) << j;
      nan |= (el & (num ^ 1u)) << j;
    }
    return pick | lowest_index<NT, E>(nan, k - n_num, J, bits, sh);
  }
  uint32_t k_rem = k - above;
  if (bsel != kNoBin && cnt_b == k_rem) {  // the whole boundary bin is taken
#pragma unroll
    for (int j = 0; j < E; ++j) pick |= (((elig >> j) & 1u) & (v[j] >= v_lo ? 1u : 0u)) << j;
    return pick;
  }
  if (bsel != kNoBin && cnt_b <= kRankMax) {
    uint32_t in_bin = 0u;
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const uint32_t el = (elig >> j) & 1u;
      const uint32_t up = v[j] >= v_hi ? 1u : 0u;
      pick |= (el & up) << j;
      in_bin |= (el & (v[j] >= v_lo ? 1u : 0u) & (up ^ 1u)) << j;
    }
    // The boundary bin's candidates go to the list, one atomic per thread.
    if (in_bin) {
      uint32_t q = atomicAdd(list_n, static_cast<uint32_t>(__popc(in_bin)));
#pragma unroll
      for (int j = 0; j < E; ++j) {
        if (!((in_bin >> j) & 1u)) continue;
        if (q < static_cast<uint32_t>(NT)) {
          list_key[q] = __float_as_uint(v[j]);
          list_idx[q] = static_cast<uint32_t>(j * NT) + threadIdx.x;
        }
        ++q;
      }
    }
    __syncthreads();
    const uint32_t m = min(*list_n, static_cast<uint32_t>(NT));
    // 2^lg threads rank one candidate (2^lg m <= NT, 2^lg <= 32, aligned
    // within a warp), each against every 2^lg-th other one, then sum over
    // those lanes. The candidates are numbers, so float order is key order.
    int lg = 5;
    while (lg > 0 && (m << lg) > static_cast<uint32_t>(NT)) --lg;
    const uint32_t cand = threadIdx.x >> lg, sub = threadIdx.x & ((1u << lg) - 1u);
    if ((threadIdx.x & ~31u) < (m << lg)) {  // warps holding a candidate
      uint32_t rank = 0u, it = 0u;
      if (cand < m) {
        const float kt = __uint_as_float(list_key[cand]);
        it = list_idx[cand];
        for (uint32_t q = sub; q < m; q += 1u << lg) {
          const float kq = __uint_as_float(list_key[q]);
          rank += (kq > kt || (kq == kt && list_idx[q] < it)) ? 1u : 0u;
        }
      }
      for (int off = (1 << lg) >> 1; off > 0; off >>= 1) rank += __shfl_xor_sync(0xffffffffu, rank, off);
      if (cand < m && sub == 0u && rank < k_rem) atomicOr(&winmap[it >> 5], 1u << (it & 31));
    }
    __syncthreads();
    if (in_bin) {
#pragma unroll
      for (int j = 0; j < E; ++j)
        if (((in_bin >> j) & 1u) && ((winmap[j * W + warp] >> lane) & 1u)) pick |= 1u << j;
    }
    return pick;
  }
  // Boundary bin too crowded (or no bin: cannot happen): exact search over
  // integer score keys. The scores turn into their keys in place (the
  // caller's array is not read after the stage), so that no second array
  // holds registers.
#pragma unroll
  for (int j = 0; j < E; ++j) v[j] = __uint_as_float(score_key(v[j]));
  uint32_t lo = 2u, hi = kTaken - 1u, cnt = n_num;
  if (bsel != kNoBin) {
    const uint32_t key_lo = score_key(v_lo), key_hi = v_hi == v_hi ? score_key(v_hi) : kTaken;
    uint32_t blo = 0xFFFFFFFFu, bhi = 0u;
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const uint32_t x = __float_as_uint(v[j]);
      if (((elig >> j) & 1u) && x >= key_lo && x < key_hi) {
        blo = min(blo, x);
        bhi = max(bhi, x);
      }
    }
    block_minmax<NT>(blo, bhi, &lo, &hi, sh);
    cnt = cnt_b;
  } else {
    k_rem = k;
  }
  for (int round = 0; round < 8; ++round) {
    if (lo == hi) break;
    const uint64_t Wd = static_cast<uint64_t>(hi - lo) + 1u;
    for (int b = threadIdx.x; b < kSelectBins; b += NT) scratch[b] = 0u;
    __syncthreads();
#pragma unroll
    for (int j = 0; j < E; ++j) {
      const uint32_t x = __float_as_uint(v[j]);
      if (((elig >> j) & 1u) && x >= lo && x <= hi)
        atomicAdd(&scratch[(static_cast<uint64_t>(x - lo) * kSelectBins) / Wd], 1u);
    }
    __syncthreads();
    uint32_t b2, above2, cnt2;
    boundary_bin<NT>(scratch, k_rem, sh, &b2, &above2, &cnt2);
    if (b2 == kNoBin) break;  // fewer candidates than k_rem: cannot happen
    k_rem -= above2;
    const uint32_t lo_b = lo + static_cast<uint32_t>((b2 * Wd + kSelectBins - 1) / kSelectBins);
    const uint32_t hi_b = lo + static_cast<uint32_t>(((b2 + 1) * Wd + kSelectBins - 1) / kSelectBins) - 1u;
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
  for (int j = 0; j < E; ++j) {
    const uint32_t el = (elig >> j) & 1u;
    const uint32_t x = __float_as_uint(v[j]);
    pick |= (el & (x > lo ? 1u : 0u)) << j;
    eq |= (el & (x == lo ? 1u : 0u)) << j;
  }
  return pick | lowest_index<NT, E>(eq, k_rem, J, bits, sh);
}

// Clears what select_slab_reg accumulates into (both histograms, both winner
// bitmaps, the list counts); needs no input, so the selection kernel runs it
// before it waits for the scores.
template <int NT, int E>
__device__ void select_reg_clear(uint32_t* smem, SelShared& sh) {
  constexpr int kWords = E * NT / 32;
  uint4* h4 = reinterpret_cast<uint4*>(smem);  // 16-byte aligned
  for (int b = threadIdx.x; b < 2 * kHistCopies * kSelectBins / 4; b += NT) h4[b] = make_uint4(0u, 0u, 0u, 0u);
  uint32_t* win = smem + 2 * kHistCopies * kSelectBins + 2 * NT;
  for (int b = threadIdx.x; b < 2 * kWords; b += NT) win[b] = 0u;
  if (threadIdx.x < 2) sh.list_cnt[threadIdx.x] = 0u;
  __syncthreads();
}

// CLEARED: the caller ran select_reg_clear on smem since its last use.
// STASH: the VaN scores wait out the TaR stage in shared memory.
template <int NT, int E, bool CLEARED = false, bool STASH = (E > kRegStashRows)>
__device__ void select_slab_reg(const SelectArgs& a, int64_t s, uint32_t* smem, SelShared& sh) {
  static_assert(E <= 32, "rows are bits of a word");
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int n_past = static_cast<int>(a.n_tokens - a.rp);
  const int J = (n_past + NT - 1) / NT;  // rows, <= E
  uint32_t* hist_t = smem;
  uint32_t* hist_v = hist_t + kHistCopies * kSelectBins;
  uint32_t* list_key = hist_v + kHistCopies * kSelectBins;
  uint32_t* list_idx = list_key + NT;
  uint32_t* win_t = list_idx + NT;
  uint32_t* win_v = win_t + E * W;
  uint32_t* bits = win_v + E * W;
  const int copy = (warp % kHistCopies) * kSelectBins;  // this warp's histogram copy
  const float* tar = a.tar + s * a.n_tokens;
  const float* van = a.van + s * a.n_tokens;
  // fma(x, sign, 0) applies the ablation's sign and turns -0 into +0 (NaN stays NaN).
  const float sgn_t = a.neg_tar ? -1.0f : 1.0f, sgn_v = a.neg_van ? -1.0f : 1.0f;
  if (!CLEARED) select_reg_clear<NT, E>(smem, sh);

  // Scores (a batch's loads issued before any is used), TaR histogram, VaN
  // range.
  float tv[E], vv[E];
  const int rows_mine = n_past > static_cast<int>(threadIdx.x) ? (n_past - 1 - static_cast<int>(threadIdx.x)) / NT + 1 : 0;
  const uint32_t mine = rows_mine >= 32 ? 0xFFFFFFFFu : ((1u << rows_mine) - 1u);
  float vmin = INFINITY, vmax = -INFINITY;  // fminf / fmaxf pass over NaN
  const Bins bt = tar_bins();
  constexpr int kB = E < 8 ? E : 8;
#pragma unroll
  for (int j0 = 0; j0 < E; j0 += kB) {
#pragma unroll
    for (int j = j0; j < j0 + kB && j < E; ++j) {
      const bool ok = (mine >> j) & 1u;
      tv[j] = ok ? __ldcg(tar + j * NT + threadIdx.x) : 0.0f;
      vv[j] = ok ? __ldcg(van + j * NT + threadIdx.x) : 0.0f;
    }
#pragma unroll
    for (int j = j0; j < j0 + kB && j < E; ++j) {
      tv[j] = fmaf(tv[j], sgn_t, 0.0f);
      vv[j] = fmaf(vv[j], sgn_v, 0.0f);
      if ((mine >> j) & 1u) {
        if (tv[j] == tv[j]) atomicAdd(&hist_t[copy + bt.of(tv[j])], 1u);
        vmin = fminf(vmin, vv[j]);
        vmax = fmaxf(vmax, vv[j]);
      }
    }
  }
  // The warps' parts of the VaN range go out with the barrier that
  // publishes the TaR histogram (nothing else writes warp_f / warp_g here).
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, off));
    vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, off));
  }
  if (lane == 0) {
    sh.warp_f[warp] = vmin;
    sh.warp_g[warp] = vmax;
  }
  __syncthreads();
  vmin = lane < W ? sh.warp_f[lane] : INFINITY;
  vmax = lane < W ? sh.warp_g[lane] : -INFINITY;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    vmin = fminf(vmin, __shfl_xor_sync(0xffffffffu, vmin, off));
    vmax = fmaxf(vmax, __shfl_xor_sync(0xffffffffu, vmax, off));
  }
  const Bins bv = range_bins(vmin, vmax);
  float* vstash = reinterpret_cast<float*>(bits + E * W);
  if (STASH) {
#pragma unroll
    for (int j = 0; j < E; ++j)
      if ((mine >> j) & 1u) vstash[j * NT + threadIdx.x] = vv[j];
  }

  // TaR stage over all past tokens.
  const uint32_t pick_t = stage_reg<NT, E>(tv, mine, J, static_cast<uint32_t>(a.n_tar),
                                           static_cast<uint32_t>(n_past), bt, hist_t, hist_t, list_key, list_idx,
                                           &sh.list_cnt[0], win_t, bits, sh);
  if (STASH) {  // each thread reads back only what it stored
#pragma unroll
    for (int j = 0; j < E; ++j) vv[j] = ((mine >> j) & 1u) ? vstash[j * NT + threadIdx.x] : 0.0f;
  }
  // VaN histogram of the tokens TaR left.
  const uint32_t rest = mine & ~pick_t;
#pragma unroll
  for (int j = 0; j < E; ++j)
    if (((rest >> j) & 1u) && vv[j] == vv[j]) atomicAdd(&hist_v[copy + bv.of(vv[j])], 1u);
  __syncthreads();  // publishes the histogram; the TaR stage's list has been read

  // VaN stage over the past tokens TaR left.
  const uint32_t pick_v = stage_reg<NT, E>(vv, rest, J, static_cast<uint32_t>(a.n_van),
                                           static_cast<uint32_t>(n_past - a.n_tar), bv, hist_v, hist_t, list_key,
                                           list_idx, &sh.list_cnt[1], win_v, bits, sh);

  // Ascending kept indices: a pick's position is the number of picks of
  // lower index (warp w's ballot over row j is word j W + w of the picks'
  // bitmap, and word order is index order), so each row's picks of a warp
  // are stored to consecutive positions; the recent frames follow.
  const uint32_t pick = pick_t | pick_v;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const uint32_t b = __ballot_sync(0xffffffffu, (pick >> j) & 1u);
    if (j < J && lane == 0) bits[j * W + warp] = b;
  }
  __syncthreads();
  const uint32_t word = static_cast<int>(threadIdx.x) < J * W ? bits[threadIdx.x] : 0u;
  uint32_t total;
  const uint32_t before = block_excl_scan<NT>(__popc(word), &total, sh);
  if (static_cast<int>(threadIdx.x) < J * W) win_t[threadIdx.x] = before;  // the TaR winners are read
  __syncthreads();
  // total == n_tar + n_van and total + rp == budget by construction; the
  // bounds only keep a broken count from writing outside this slab's row.
  int32_t* kept = a.kept + s * a.budget;
  const uint32_t lt = (1u << lane) - 1u;
#pragma unroll
  for (int j = 0; j < E; ++j) {
    const uint32_t b = __ballot_sync(0xffffffffu, (pick >> j) & 1u);
    if ((pick >> j) & 1u) {
      const uint32_t at = win_t[j * W + warp] + __popc(b & lt);
      if (at < a.budget) kept[at] = static_cast<int32_t>(j * NT + threadIdx.x);
    }
  }
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
// coalesced (ids travel with their rows, Sec. 3.1 K~ = K[:, I, :]). A
// thread's kB elements are loaded together (kept indices, then the ids they
// point to), so it waits for two round trips per batch, not two per element.
__device__ __forceinline__ void gather_ids(const GatherArgs& a) {
  if (!a.pid_dst && !a.fid_dst) return;
  constexpr int kB = 4;
  const int64_t total = a.n_slabs * a.budget;
  const int64_t step = static_cast<int64_t>(gridDim.x) * blockDim.x;
  for (int64_t g0 = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; g0 < total; g0 += kB * step) {
    int n[kB];
    int64_t base[kB], j[kB];
#pragma unroll
    for (int u = 0; u < kB; ++u) {
      const int64_t g = g0 + u * step;
      n[u] = -1;
      base[u] = 0;
      j[u] = 0;
      if (g < total) {
        const int64_t s = g / a.budget;
        j[u] = g - s * a.budget;
        base[u] = s * a.cap;
        n[u] = a.heads_per_kept > 1 ? a.kept[(s / a.heads_per_kept) * a.budget + j[u]] : a.kept[g];
      }
    }
    uint16_t pv[kB];
    uint32_t fv[kB];
#pragma unroll
    for (int u = 0; u < kB; ++u) {
      const bool ok = n[u] >= 0 && n[u] < a.cap;
      pv[u] = 0;
      fv[u] = 0;
      if (ok && a.pid_dst) pv[u] = a.pid_src ? a.pid_src[base[u] + n[u]] : static_cast<uint16_t>(n[u] % a.p);
      if (ok && a.fid_dst) fv[u] = a.fid_src ? a.fid_src[base[u] + n[u]] : static_cast<uint32_t>(n[u] / a.p);
    }
#pragma unroll
    for (int u = 0; u < kB; ++u) {
      if (n[u] < 0 || n[u] >= a.cap) continue;
      if (a.pid_dst) a.pid_dst[base[u] + j[u]] = pv[u];
      if (a.fid_dst) a.fid_dst[base[u] + j[u]] = fv[u];
    }
  }
}

}  // namespace dev
}  // namespace ipv
