// Device building blocks of the compression pass, shared by the staged
// kernels (score.cu, select.cu, gather.cu) and the single-kernel pipeline
// (pipeline.cu), so that both paths run exactly the same arithmetic.
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

// TaR and VaN of past rows [lo, hi) of slab s by every warp of the block
// (block-uniform arguments). Sec. 3.1 Eq. (tar): s_TaR = -(k . m_q) / max(|k|, eps);
// Sec. 3.2: s_VaN = |v|. Each warp step covers 32/LPR consecutive rows; kU
// steps are loaded before any is reduced. mtab rows are ms floats apart.
template <typename T, int LPR, int CPL, int kU, int MSRC>
__device__ __forceinline__ void score_segment(const ScoreArgs& a, int64_t s, int lo, int hi,
                                              const float* mtab, int ms) {
  constexpr int E = Chunk<T>::kElems;
  constexpr int P2 = Chunk<T>::kPairs;
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
      const float dot = group_sum<LPR>(dot2.x + dot2.y);
      const float kk = group_sum<LPR>(kk2.x + kk2.y);
      const float vv = group_sum<LPR>(vv2.x + vv2.y);
      if (sub == 0 && n < hi) {
        // max(|k|, eps) = sqrt(max(|k|^2, eps^2)). A patch id outside [0, p)
        // has no recent-frame partner: NaN scores rank below every number,
        // so such a token is never preferred.
        if (a.kk) {  // the shared index set: this head's partial sums
          tar[n] = q_ok ? dot : __int_as_float(0x7fc00000);
          a.kk[s * a.n_tokens + n] = kk;
          van[n] = q_ok ? vv : __int_as_float(0x7fc00000);
        } else {
          tar[n] = q_ok ? -dot * rsqrtf(fmaxf(kk, kNormEps * kNormEps)) : __int_as_float(0x7fc00000);
          van[n] = q_ok ? sqrtf(vv) : __int_as_float(0x7fc00000);
        }
      }
    }
    q_base += step_mod;
    q_base = q_base >= p ? q_base - p : q_base;
  }
}

// Shared-memory bookkeeping of the bulk-copy ring (static, per block).
struct BulkRing {
  uint64_t full[kMaxStages];    // completes when a stage's copies have landed
  unsigned done[kMaxStages];    // warps finished with the stage's current chunk
  unsigned issued[kMaxStages];  // copies ever issued into the stage
};

__device__ __forceinline__ void ring_init(BulkRing& rg, int nst) {  // thread 0
  for (int i = 0; i < nst; ++i) {
    mbar_init(&rg.full[i], 1u);
    rg.done[i] = 0u;
    rg.issued[i] = 0u;
  }
  mbar_init_fence();
}

// Copies a slab's m table ([p][D] fp32, global) into shared memory in the
// layout score_segment_bulk reads: each row split into E/4 planes, plane j
// holding floats 4j..4j+3 of every 16-byte chunk of K (E elements per chunk),
// so the lanes of a row read 16 consecutive bytes each. RO: the table is not
// written by the running kernel (read through the non-coherent path).
template <typename T, bool RO>
__device__ __forceinline__ void load_m_planes(const float* m_slab, float* m_tab, int p, int D) {
  constexpr int kPlanes = Chunk<T>::kElems / 4;
  const int d4 = D / 4;  // float4s per row
  const float4* src = reinterpret_cast<const float4*>(m_slab);
  float4* dst = reinterpret_cast<float4*>(m_tab);
  for (int i = threadIdx.x; i < p * d4; i += blockDim.x) {
    const int q = i / d4, f = i - q * d4;
    const int c = f / kPlanes, pl = f - c * kPlanes;
    dst[q * d4 + pl * (d4 / kPlanes) + c] = RO ? __ldg(src + i) : src[i];
  }
}

// Bulk-copy-fed version of score_segment. A ring of nst stages, each R
// consecutive rows of K followed by the same rows of V (R = all warps' rows of
// one warp step, 16 KB per copy at the usual shapes), is filled by cp.async.bulk.
// Warps consume every stage independently and count themselves out; the warp
// that finishes a stage last refills it with the chunk nst steps ahead, so no
// block-wide barrier is taken while streaming and copies stay large. 8/16/32
// lanes share a row: a shared-memory phase reads one row's 128 contiguous
// bytes (no bank conflicts). m_tab is the slab's m table in shared memory in
// the layout of load_m_planes; seq counts the stages this block has used (barrier parity) and is
// kept by the caller across segments. On a barrier timeout the warp stops,
// sets bit 2 of *a.error, and the block drains its copies before returning.
template <typename T, int LPR, int CPL>
__device__ __forceinline__ void score_segment_bulk(const ScoreArgs& a, int64_t s, int lo, int hi,
                                                   const float* m_tab, char* stages, int nst,
                                                   BulkRing& rg, uint32_t& seq) {
  constexpr int P2 = Chunk<T>::kPairs;
  constexpr int kPlanes = Chunk<T>::kElems / 4;
  constexpr int RPW = 32 / LPR;
  const int lane = threadIdx.x & 31;
  const int sub = lane % LPR, grp = lane / LPR;
  const int warp = threadIdx.x >> 5, n_warps = blockDim.x >> 5;
  const int row_bytes = a.D * static_cast<int>(sizeof(T));
  const int n_chunks = row_bytes / 16;
  const int R = n_warps * RPW;
  const int stage_bytes = 2 * R * row_bytes;
  const int p = a.p;
  const char* kslab = static_cast<const char*>(a.k) + s * a.cap * row_bytes;
  const char* vslab = static_cast<const char*>(a.v) + s * a.cap * row_bytes;
  const uint16_t* pid = a.patch_id ? a.patch_id + s * a.cap : nullptr;
  float* tar = a.tar + s * a.n_tokens;
  float* van = a.van + s * a.n_tokens;
  const int n_steps = (hi - lo + R - 1) / R;
  const int my_row = warp * RPW + grp;
  const uint32_t seq0 = seq;

  auto issue = [&](int j) {  // one thread
    const uint32_t slot = (seq0 + j) % nst;
    const int r0 = lo + j * R;
    const uint32_t bytes = static_cast<uint32_t>(min(R, hi - r0) * row_bytes);
    char* dst = stages + slot * stage_bytes;
    fence_proxy_async_smem();  // earlier ordinary accesses to this stage come first
    rg.issued[slot] += 1u;
    mbar_expect_tx(&rg.full[slot], 2u * bytes);
    bulk_g2s(dst, kslab + static_cast<int64_t>(r0) * row_bytes, bytes, &rg.full[slot]);
    bulk_g2s(dst + R * row_bytes, vslab + static_cast<int64_t>(r0) * row_bytes, bytes, &rg.full[slot]);
  };
  if (threadIdx.x == 0)
    for (int j = 0; j < nst && j < n_steps; ++j) issue(j);

  int j = 0;
  for (; j < n_steps; ++j) {
    const uint32_t slot = (seq0 + j) % nst;
    const bool landed = mbar_wait(&rg.full[slot], ((seq0 + j) / nst) & 1u);
    if (__any_sync(0xffffffffu, !landed)) break;
    const char* kst = stages + slot * stage_bytes + my_row * row_bytes;
    const char* vst = kst + R * row_bytes;
    const int n = lo + j * R + my_row;
    const bool ok = n < hi;
    const int q = pid ? (ok ? static_cast<int>(pid[n]) : 0) : n % p;
    const bool q_ok = q < p;
    const float* mq = m_tab + (q_ok ? q : 0) * a.D;
    float2 dot2 = make_float2(0.0f, 0.0f), kk2 = dot2, vv2 = dot2;
#pragma unroll
    for (int k = 0; k < CPL; ++k) {
      const int c = sub + LPR * k;
      if (ok && c < n_chunks) {
        float2 kx[P2], vx[P2];
        Chunk<T>::widen2(*reinterpret_cast<const uint4*>(kst + c * 16), kx);
        Chunk<T>::widen2(*reinterpret_cast<const uint4*>(vst + c * 16), vx);
#pragma unroll
        for (int e = 0; e < P2; e += 2) {
          // m_tab row layout: plane e/2 holds floats 2e..2e+3 of every chunk.
          const float4 mv = *reinterpret_cast<const float4*>(mq + (e / 2) * (a.D / kPlanes) + c * 4);
          dot2 = fma2(kx[e], make_float2(mv.x, mv.y), dot2);
          dot2 = fma2(kx[e + 1], make_float2(mv.z, mv.w), dot2);
        }
#pragma unroll
        for (int e = 0; e < P2; ++e) {
          kk2 = fma2(kx[e], kx[e], kk2);
          vv2 = fma2(vx[e], vx[e], vv2);
        }
      }
    }
    const float dot = group_sum<LPR>(dot2.x + dot2.y);
    const float kk = group_sum<LPR>(kk2.x + kk2.y);
    const float vv = group_sum<LPR>(vv2.x + vv2.y);
    if (sub == 0 && ok) {
      // max(|k|, eps) = sqrt(max(|k|^2, eps^2)). A patch id outside [0, p)
      // has no recent-frame partner: NaN scores rank below every number.
      tar[n] = q_ok ? -dot * rsqrtf(fmaxf(kk, kNormEps * kNormEps)) : __int_as_float(0x7fc00000);
      van[n] = q_ok ? sqrtf(vv) : __int_as_float(0x7fc00000);
    }
    __syncwarp();
    if (lane == 0) {
      __threadfence_block();  // this warp's reads of the stage are done
      if (atomicAdd(&rg.done[slot], 1u) == static_cast<unsigned>(n_warps - 1)) {
        rg.done[slot] = 0u;  // last warp out: refill the stage
        __threadfence_block();
        if (j + nst < n_steps) issue(j + nst);
      }
    }
  }
  seq = seq0 + n_steps;
  if (__syncthreads_or(j < n_steps)) {  // a barrier timed out somewhere
    if (threadIdx.x == 0) {
      atomicOr(a.error, 4u);
      for (int k = 0; k < nst; ++k)  // wait for the last copy issued into each stage
        if (rg.issued[k]) mbar_wait(&rg.full[k], (rg.issued[k] - 1u) & 1u);
      for (int k = 0; k < nst; ++k) rg.done[k] = 0u;
    }
    __syncthreads();
  }
}

// ------------------------------------------------------------------ selection
// Per slab (Sec. 3.3; Algorithm 1 steps 3-5): keep the r p recent tokens,
// take the n_tar past tokens of highest s_TaR, then the n_van past tokens of
// highest s_VaN among those TaR left (Algorithm 2's max-forcing of TaR picks
// before its final TopK). Ties go to the lower index; NaN ranks lowest.
//
// One block of NT threads per slab; scores live in shared memory as
// order-preserving uint32 keys. A stage finds its k winners without a sort: a
// 2048-bin histogram linear in the score value over [min, max] of the
// candidates (a monotone map, so every bin above the one holding the k-th
// winner is taken whole); the candidates of that boundary bin are ranked
// exactly against each other with the index tie-break. A boundary bin of
// more than NT candidates falls back to an exact search over integer key
// windows with ties counted by a block-wide prefix sum in index order.
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

// Shared memory of select_slab: keys[pad4(n_past)], hist[2048], list_key[NT],
// list_idx[NT], and with a.van_smem the VaN scores[pad4(n_past)].
template <int NT>
__host__ __device__ constexpr size_t select_smem_words(int64_t n_past, bool van_smem = false) {
  return static_cast<size_t>((n_past + 3) & ~3LL) * (van_smem ? 2 : 1) + kSelectBins + 2 * NT;
}

__device__ __forceinline__ bool is_cand(uint32_t k) { return k != kExcluded && k != kTaken; }

__device__ __forceinline__ float key_value(uint32_t k) {  // inverse of score_key, keys >= 2
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

__device__ __forceinline__ int value_bin(float v, float vmin, float scale) {  // monotone
  const int b = static_cast<int>((v - vmin) * scale);
  return b < kSelectBins - 1 ? b : kSelectBins - 1;
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

struct Stats {  // value range and NaN count of a stage's candidates
  float vmin, vmax;
  uint32_t n_nan;
};

__device__ __forceinline__ void stats_add(Stats& st, float v) {
  if (v != v) {
    ++st.n_nan;
  } else {
    st.vmin = fminf(st.vmin, v);
    st.vmax = fmaxf(st.vmax, v);
  }
}

template <int NT>
__device__ Stats block_stats(Stats st, SelShared& sh) {
  constexpr int W = NT / 32;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    st.vmin = fminf(st.vmin, __shfl_xor_sync(0xffffffffu, st.vmin, off));
    st.vmax = fmaxf(st.vmax, __shfl_xor_sync(0xffffffffu, st.vmax, off));
    st.n_nan += __shfl_xor_sync(0xffffffffu, st.n_nan, off);
  }
  if (lane == 0) {
    sh.warp_f[warp] = st.vmin;
    sh.warp_g[warp] = st.vmax;
    sh.warp_a[warp] = st.n_nan;
  }
  __syncthreads();
  if (warp == 0) {
    st.vmin = lane < W ? sh.warp_f[lane] : INFINITY;
    st.vmax = lane < W ? sh.warp_g[lane] : -INFINITY;
    st.n_nan = lane < W ? sh.warp_a[lane] : 0u;
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      st.vmin = fminf(st.vmin, __shfl_xor_sync(0xffffffffu, st.vmin, off));
      st.vmax = fmaxf(st.vmax, __shfl_xor_sync(0xffffffffu, st.vmax, off));
      st.n_nan += __shfl_xor_sync(0xffffffffu, st.n_nan, off);
    }
    if (lane == 0) {
      sh.fcast[0] = st.vmin;
      sh.fcast[1] = st.vmax;
      sh.bcast[0] = st.n_nan;
    }
  }
  __syncthreads();
  Stats out{sh.fcast[0], sh.fcast[1], sh.bcast[0]};
  __syncthreads();
  return out;
}

// The bin holding the k-th largest candidate (bins scanned from the top;
// thread t owns the 2048/NT bins just below bin 2048 - t 2048/NT), the count
// of candidates in higher bins and the bin's own count. kNoBin if the
// histogram holds fewer than k.
template <int NT>
__device__ void boundary_bin(const uint32_t* hist, uint32_t k, SelShared& sh, uint32_t* bsel,
                             uint32_t* above, uint32_t* cnt_b) {
  constexpr int BPT = kSelectBins / NT;
  const int top = kSelectBins - 1 - BPT * static_cast<int>(threadIdx.x);
  uint32_t h[BPT], local = 0u;
#pragma unroll
  for (int j = 0; j < BPT; ++j) {
    h[j] = hist[top - j];
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
// The window shrinks at least 2048-fold per round (4 rounds for 32-bit
// keys); the hard round limit only guards against a broken invariant.
template <int NT>
__device__ void window_search(const uint32_t* key, int n, uint32_t lo, uint32_t hi, uint32_t k,
                              uint32_t cnt, uint32_t* hist, SelShared& sh, uint32_t* T,
                              uint32_t* take_eq, uint32_t* cnt_eq) {
  for (int round = 0; round < 8; ++round) {
    if (lo == hi) break;
    const uint64_t W = static_cast<uint64_t>(hi - lo) + 1u;
    for (int b = threadIdx.x; b < kSelectBins; b += NT) hist[b] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += NT) {
      const uint32_t x = key[i];
      if (x >= lo && x <= hi)
        atomicAdd(&hist[(static_cast<uint64_t>(x - lo) * kSelectBins) / W], 1u);
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
  int mode;  // 0 none, 1 every candidate, 2 key threshold, 3 value bin (+ pre-marked)
  uint32_t T, take, cnt_eq;
  int bthr;
  float vmin, scale;
};

// Decides a stage taking the k best of n_cand candidates. Boundary-bin
// winners found by direct ranking are marked in place with `mark`.
template <int NT>
__device__ Plan plan_stage(uint32_t* key, int n, uint32_t k, uint32_t n_cand, Stats st,
                           uint32_t mark, uint32_t* hist, uint32_t* list_key, uint32_t* list_idx,
                           SelShared& sh) {
  Plan P{};
  if (k == 0u) return P;
  if (k >= n_cand) {
    P.mode = 1;
    return P;
  }
  const uint32_t n_num = n_cand - st.n_nan;
  P.mode = 2;
  if (k > n_num) {  // every number, then the lowest-index NaNs
    P.T = kNanKey;
    P.take = k - n_num;
    P.cnt_eq = st.n_nan;
    return P;
  }
  if (st.vmin == st.vmax) {  // all numbers equal
    P.T = score_key(st.vmin);
    P.take = k;
    P.cnt_eq = n_num;
    return P;
  }
  const float range = st.vmax - st.vmin;
  const float scale = static_cast<float>(kSelectBins) / range;
  uint32_t lo = score_key(st.vmin), hi = score_key(st.vmax), k_rem = k, cnt = n_num;
  if (range < INFINITY && scale < INFINITY) {
    for (int b = threadIdx.x; b < kSelectBins; b += NT) hist[b] = 0u;
    if (threadIdx.x == 0) sh.list_n = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += NT) {
      const uint32_t x = key[i];
      if (is_cand(x) && x != kNanKey) atomicAdd(&hist[value_bin(key_value(x), st.vmin, scale)], 1u);
    }
    __syncthreads();
    uint32_t bsel, above, cnt_b;
    boundary_bin<NT>(hist, k, sh, &bsel, &above, &cnt_b);
    if (bsel != kNoBin) {
      k_rem = k - above;
      P.mode = 3;
      P.vmin = st.vmin;
      P.scale = scale;
      if (cnt_b == k_rem) {  // the whole boundary bin is taken
        P.bthr = static_cast<int>(bsel) - 1;
        return P;
      }
      P.bthr = static_cast<int>(bsel);
      if (cnt_b <= static_cast<uint32_t>(NT)) {
        for (int i = threadIdx.x; i < n; i += NT) {
          const uint32_t x = key[i];
          if (is_cand(x) && x != kNanKey &&
              value_bin(key_value(x), st.vmin, scale) == static_cast<int>(bsel)) {
            const uint32_t j = atomicAdd(&sh.list_n, 1u);
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
        if (is_cand(x) && x != kNanKey &&
            value_bin(key_value(x), st.vmin, scale) == static_cast<int>(bsel)) {
          blo = min(blo, x);
          bhi = max(bhi, x);
        }
      }
      block_minmax<NT>(blo, bhi, &lo, &hi, sh);
      cnt = cnt_b;
    }
  }
  P.mode = 2;
  window_search<NT>(key, n, lo, hi, k_rem, cnt, hist, sh, &P.T, &P.take, &P.cnt_eq);
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
      case 3: return x != kNanKey && value_bin(key_value(x), P.vmin, P.scale) > P.bthr;
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
// select_smem_words<NT>(n_past) words. Scores are read with plain loads (they
// may have been written earlier in the same kernel).
template <int NT>
__device__ void select_slab(const SelectArgs& a, int64_t s, uint32_t* smem, SelShared& sh) {
  const int n_past = static_cast<int>(a.n_tokens - a.rp);
  uint32_t* key = smem;
  uint32_t* hist = smem + ((n_past + 3) & ~3);
  uint32_t* list_key = hist + kSelectBins;
  uint32_t* list_idx = list_key + NT;
  const float* tar = a.tar + s * a.n_tokens;
  const float* van = a.van + s * a.n_tokens;
  const int chunk = (n_past + NT - 1) / NT;
  const int c0 = min(n_past, static_cast<int>(threadIdx.x) * chunk);
  const int c1 = min(n_past, c0 + chunk);

  // VaN goes to shared memory in the same pass as TaR when there is room,
  // so that the VaN stage does not wait for a second round of loads.
  float* vbuf = a.van_smem ? reinterpret_cast<float*>(list_idx + NT) : nullptr;

  // TaR stage over all past tokens.
  Stats st{INFINITY, -INFINITY, 0u};
  for (int i = threadIdx.x; i < n_past; i += NT) {
    const float v = (a.neg_tar ? -tar[i] : tar[i]) + 0.0f;  // NaN stays NaN, -0 becomes +0
    if (vbuf) vbuf[i] = van[i];
    key[i] = score_key(v);
    stats_add(st, v);
  }
  st = block_stats<NT>(st, sh);
  Plan P = plan_stage<NT>(key, n_past, static_cast<uint32_t>(a.n_tar), static_cast<uint32_t>(n_past),
                          st, kExcluded, hist, list_key, list_idx, sh);
  Picker pk = make_picker<NT>(key, c0, c1, P, kExcluded, sh);
  Stats sv{INFINITY, -INFINITY, 0u};
  for (int i0 = c0; i0 < c1; i0 += 8) {
    float vb[8];  // issue the VaN loads of 8 tokens before using any
#pragma unroll
    for (int b = 0; b < 8; ++b) vb[b] = (i0 + b < c1) ? (vbuf ? vbuf[i0 + b] : van[i0 + b]) : 0.0f;
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const int i = i0 + b;
      if (i >= c1) break;
      if (pk.pick(key[i])) {
        key[i] = kExcluded;
      } else {
        const float v = (a.neg_van ? -vb[b] : vb[b]) + 0.0f;
        key[i] = score_key(v);
        stats_add(sv, v);
      }
    }
  }
  sv = block_stats<NT>(sv, sh);  // its barriers also publish the keys

  // VaN stage over the past tokens TaR left.
  const uint32_t n_rest = static_cast<uint32_t>(n_past - a.n_tar);
  P = plan_stage<NT>(key, n_past, static_cast<uint32_t>(a.n_van), n_rest, sv, kTaken, hist,
                     list_key, list_idx, sh);
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
}

// ------------------------------------------------------------------ compaction
// Sec. 3.1 / Algorithm 2 last step: dst row j of a slab = src row kept[j].
// Half-warp hw (of n_hw) copies rows g = g_begin + hw, g_begin + hw + n_hw,
// ... of the flattened (slab, j) range [g_begin, g_end), kU rows in flight.
// Kept indices and source patch ids are read with plain loads (the kept
// indices may have been written earlier in the same kernel). IDS: copy the
// patch and frame ids of each row here too (else gather_ids does it).
// JN > 0 (the step kernels): g runs over (slab, j) with j < jn kept rows per
// slab, the kept stride staying a.budget; FIXED: the source row is
// a.n_tokens - a.rp + j and kept is not read (the recent frames, j < rp,
// written to rows budget - rp + j).
template <int CPL, int kU, bool IDS = true, bool FIXED = false>
__device__ __forceinline__ void gather_range(const GatherArgs& a, int64_t g_begin, int64_t g_end,
                                             int64_t hw, int64_t n_hw, int64_t jn = 0) {
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
          n = a.kept[(a.heads_per_kept > 1 ? s / a.heads_per_kept : s) * a.budget + j];
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
        kr[u][c] = ld ? ld_stream(ks + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
        vr[u][c] = ld ? ld_stream(vs + src_off + ch * 16) : make_uint4(0, 0, 0, 0);
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
