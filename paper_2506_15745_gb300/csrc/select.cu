// Step (iii) of the compression pass: the split-budget selection.
//
// Per (layer, KV head) slab (InfiniPot-V Sec. 3.3; Algorithm 1 steps 3-5):
// the r*p recent tokens are kept; the n_tar past tokens of highest s_TaR are
// taken; then the n_van past tokens of highest s_VaN among those TaR left
// (Algorithm 2 forces TaR picks to max(VaN) before its final TopK, which is
// the same as excluding them). Ties go to the lower token index; NaN ranks
// below every number. The kept set is written as ascending row indices.
//
// One 1024-thread CTA per slab; scores live in shared memory as
// order-preserving uint32 keys. Each stage finds its k winners without a
// sort: a 2048-bin histogram that is linear in the score value over
// [min, max] of the candidates (a monotone map, so every bin above the one
// holding the k-th winner is taken whole); the candidates of that boundary
// bin, usually a few dozen, are ranked exactly against each other with the
// index tie-break. A boundary bin of more than 1024 candidates (heavy ties
// or extreme clustering) falls back to an exact search over integer key
// windows with ties counted by a block-wide prefix sum in index order.
#include "ipv_common.cuh"

namespace ipv {
namespace {

constexpr uint32_t kTaken = 0xFFFFFFFFu;    // VaN pick (never a score key)
constexpr uint32_t kExcluded = 0u;          // TaR pick, excluded from the VaN stage
constexpr uint32_t kNanKey = 1u;            // score_key of every NaN
constexpr uint32_t kNoBin = 0xFFFFFFFFu;
constexpr int kListMax = kSelectThreads;    // boundary candidates ranked directly

struct BlockShared {
  uint32_t warp_a[32];
  uint32_t warp_b[32];
  float warp_f[32];
  float warp_g[32];
  uint32_t bcast[8];
  float fcast[2];
  uint32_t list_n;
};

// Candidates of a stage: real score keys (NaN included), not yet taken.
__device__ __forceinline__ bool is_cand(uint32_t k) { return k != kExcluded && k != kTaken; }

// Inverse of score_key for keys >= 2.
__device__ __forceinline__ float key_value(uint32_t k) {
  return __uint_as_float((k & 0x80000000u) ? (k & 0x7FFFFFFFu) : ~k);
}

// Monotone non-decreasing bin of a score in [vmin, vmax].
__device__ __forceinline__ int value_bin(float v, float vmin, float scale) {
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

// Exclusive prefix sum over the 1024 threads in thread order; *total gets the sum.
__device__ uint32_t block_excl_scan(uint32_t v, uint32_t* total, BlockShared& sh) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const uint32_t incl = warp_incl_scan(v);
  if (lane == 31) sh.warp_a[warp] = incl;
  __syncthreads();
  if (warp == 0) {
    const uint32_t w = sh.warp_a[lane];
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

// Block-wide min/max of uint32 keys; broadcast to all threads.
__device__ void block_minmax(uint32_t lo, uint32_t hi, uint32_t* out_lo, uint32_t* out_hi,
                             BlockShared& sh) {
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
    lo = sh.warp_a[lane];
    hi = sh.warp_b[lane];
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

// Value range and NaN count of a stage's candidates.
struct Stats {
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

__device__ Stats block_stats(Stats st, BlockShared& sh) {
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
    st.vmin = sh.warp_f[lane];
    st.vmax = sh.warp_g[lane];
    st.n_nan = sh.warp_a[lane];
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

// Finds, from the histogram, the bin holding the k-th largest candidate
// (bins scanned from the top). Thread t owns bins 2047-2t and 2046-2t.
// Returns the bin (kNoBin if the histogram holds fewer than k), the count of
// candidates in higher bins and the bin's own count.
__device__ void boundary_bin(const uint32_t* hist, uint32_t k, BlockShared& sh, uint32_t* bsel,
                             uint32_t* above, uint32_t* cnt_b) {
  const int ba = kSelectBins - 1 - 2 * static_cast<int>(threadIdx.x), bb = ba - 1;
  const uint32_t ha = hist[ba], hb = hist[bb];
  if (threadIdx.x == 0) sh.bcast[2] = kNoBin;  // published by the scan's barriers
  uint32_t tot;
  const uint32_t above_a = block_excl_scan(ha + hb, &tot, sh);
  const uint32_t above_b = above_a + ha;
  if (above_a < k && k <= above_a + ha) {
    sh.bcast[2] = ba;
    sh.bcast[3] = above_a;
    sh.bcast[4] = ha;
  } else if (above_b < k && k <= above_b + hb) {
    sh.bcast[2] = bb;
    sh.bcast[3] = above_b;
    sh.bcast[4] = hb;
  }
  __syncthreads();
  *bsel = sh.bcast[2];
  *above = sh.bcast[3];
  *cnt_b = sh.bcast[4];
  __syncthreads();
}

// Exact threshold search over integer key windows, starting from the window
// [lo, hi] that holds cnt candidates of which the k largest are wanted (all
// candidates above hi are taken already). On return the winners are the
// candidates with key > *T plus the *take lowest-index ones with key == *T;
// *cnt_eq counts the candidates equal to *T. The window shrinks at least
// 2048-fold per round (4 rounds for 32-bit keys); the hard round limit only
// guards against a broken invariant.
__device__ void window_search(const uint32_t* key, int n, uint32_t lo, uint32_t hi, uint32_t k,
                              uint32_t cnt, uint32_t* hist, BlockShared& sh, uint32_t* T,
                              uint32_t* take_eq, uint32_t* cnt_eq) {
  for (int round = 0; round < 8; ++round) {
    if (lo == hi) break;
    const uint64_t W = static_cast<uint64_t>(hi - lo) + 1u;
    for (int b = threadIdx.x; b < kSelectBins; b += kSelectThreads) hist[b] = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += kSelectThreads) {
      const uint32_t x = key[i];
      if (x >= lo && x <= hi)
        atomicAdd(&hist[(static_cast<uint64_t>(x - lo) * kSelectBins) / W], 1u);
    }
    __syncthreads();
    uint32_t bsel, above, cnt_b;
    boundary_bin(hist, k, sh, &bsel, &above, &cnt_b);
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
__device__ Plan plan_stage(uint32_t* key, int n, uint32_t k, uint32_t n_cand, Stats st,
                           uint32_t mark, uint32_t* hist, uint32_t* list_key, uint32_t* list_idx,
                           BlockShared& sh) {
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
    for (int b = threadIdx.x; b < kSelectBins; b += kSelectThreads) hist[b] = 0u;
    if (threadIdx.x == 0) sh.list_n = 0u;
    __syncthreads();
    for (int i = threadIdx.x; i < n; i += kSelectThreads) {
      const uint32_t x = key[i];
      if (is_cand(x) && x != kNanKey) atomicAdd(&hist[value_bin(key_value(x), st.vmin, scale)], 1u);
    }
    __syncthreads();
    uint32_t bsel, above, cnt_b;
    boundary_bin(hist, k, sh, &bsel, &above, &cnt_b);
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
      if (cnt_b <= static_cast<uint32_t>(kListMax)) {
        for (int i = threadIdx.x; i < n; i += kSelectThreads) {
          const uint32_t x = key[i];
          if (is_cand(x) && x != kNanKey &&
              value_bin(key_value(x), st.vmin, scale) == static_cast<int>(bsel)) {
            const uint32_t j = atomicAdd(&sh.list_n, 1u);
            if (j < static_cast<uint32_t>(kListMax)) {
              list_key[j] = x;
              list_idx[j] = static_cast<uint32_t>(i);
            }
          }
        }
        __syncthreads();
        const uint32_t m = min(sh.list_n, static_cast<uint32_t>(kListMax));
        if (threadIdx.x < m) {
          const uint32_t kt = list_key[threadIdx.x], it = list_idx[threadIdx.x];
          uint32_t rank = 0u;
          for (uint32_t j = 0; j < m; ++j) {
            const uint32_t kj = list_key[j];
            rank += (kj > kt || (kj == kt && list_idx[j] < it)) ? 1u : 0u;
          }
          if (rank < k_rem) key[it] = mark;
        }
        __syncthreads();
        return P;
      }
      // Too many candidates in the bin: exact search inside its key range.
      uint32_t blo = 0xFFFFFFFFu, bhi = 0u;
      for (int i = threadIdx.x; i < n; i += kSelectThreads) {
        const uint32_t x = key[i];
        if (is_cand(x) && x != kNanKey &&
            value_bin(key_value(x), st.vmin, scale) == static_cast<int>(bsel)) {
          blo = min(blo, x);
          bhi = max(bhi, x);
        }
      }
      block_minmax(blo, bhi, &lo, &hi, sh);
      cnt = cnt_b;
    }
  }
  P.mode = 2;
  window_search(key, n, lo, hi, k_rem, cnt, hist, sh, &P.T, &P.take, &P.cnt_eq);
  return P;
}

// Rank-among-ties bookkeeping: each thread walks the contiguous chunk
// [c0, c1) of indices; returns the number of keys equal to T in the chunks of
// lower-numbered threads.
__device__ uint32_t ties_before(const uint32_t* key, int c0, int c1, uint32_t T, BlockShared& sh) {
  uint32_t mine = 0u;
  for (int i = c0; i < c1; ++i) mine += (key[i] == T) ? 1u : 0u;
  uint32_t tot;
  return block_excl_scan(mine, &tot, sh);
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

__device__ Picker make_picker(const uint32_t* key, int c0, int c1, const Plan& P, uint32_t mark,
                              BlockShared& sh) {
  Picker pk{P, mark, 0u, true};
  if (P.mode == 2 && P.take > 0u && P.take < P.cnt_eq) {
    pk.all_ties = false;
    pk.rank = ties_before(key, c0, c1, P.T, sh);
  } else if (P.mode == 2 && P.take == 0u) {
    pk.all_ties = false;  // nothing equal to T is taken
  }
  return pk;
}

__global__ void __launch_bounds__(kSelectThreads, 1) select_kernel(SelectArgs a) {
  extern __shared__ uint32_t sm_key[];
  __shared__ BlockShared sh;
  __shared__ uint32_t list_key[kListMax];
  __shared__ uint32_t list_idx[kListMax];
  const int n_past = static_cast<int>(a.n_tokens - a.rp);
  uint32_t* key = sm_key;
  uint32_t* hist = sm_key + ((n_past + 3) & ~3);
  const int64_t s = blockIdx.x;
  const float* tar = a.tar + s * a.n_tokens;
  const float* van = a.van + s * a.n_tokens;
  const int chunk = (n_past + kSelectThreads - 1) / kSelectThreads;
  const int c0 = min(n_past, static_cast<int>(threadIdx.x) * chunk);
  const int c1 = min(n_past, c0 + chunk);

  // TaR stage over all past tokens.
  Stats st{INFINITY, -INFINITY, 0u};
  for (int i = threadIdx.x; i < n_past; i += kSelectThreads) {
    const float v = tar[i] + 0.0f;
    key[i] = score_key(v);
    stats_add(st, v);
  }
  st = block_stats(st, sh);
  Plan P = plan_stage(key, n_past, static_cast<uint32_t>(a.n_tar), static_cast<uint32_t>(n_past),
                      st, kExcluded, hist, list_key, list_idx, sh);
  Picker pk = make_picker(key, c0, c1, P, kExcluded, sh);
  Stats sv{INFINITY, -INFINITY, 0u};
  for (int i0 = c0; i0 < c1; i0 += 8) {
    float vb[8];  // issue the VaN loads of 8 tokens before using any
#pragma unroll
    for (int b = 0; b < 8; ++b) vb[b] = (i0 + b < c1) ? van[i0 + b] : 0.0f;
#pragma unroll
    for (int b = 0; b < 8; ++b) {
      const int i = i0 + b;
      if (i >= c1) break;
      if (pk.pick(key[i])) {
        key[i] = kExcluded;
      } else {
        const float v = vb[b] + 0.0f;
        key[i] = score_key(v);
        stats_add(sv, v);
      }
    }
  }
  sv = block_stats(sv, sh);  // its barriers also publish the keys

  // VaN stage over the past tokens TaR left.
  const uint32_t n_rest = static_cast<uint32_t>(n_past - a.n_tar);
  P = plan_stage(key, n_past, static_cast<uint32_t>(a.n_van), n_rest, sv, kTaken, hist, list_key,
                 list_idx, sh);
  pk = make_picker(key, c0, c1, P, kTaken, sh);
  for (int i = c0; i < c1; ++i)
    if (pk.pick(key[i])) key[i] = kTaken;
  __syncthreads();

  // Ascending kept indices: past picks, then the recent frames.
  uint32_t mine = 0u;
  for (int i = c0; i < c1; ++i) mine += (key[i] == kExcluded || key[i] == kTaken) ? 1u : 0u;
  uint32_t total;
  uint32_t pos = block_excl_scan(mine, &total, sh);
  int32_t* kept = a.kept + s * a.budget;
  for (int i = c0; i < c1; ++i)
    if ((key[i] == kExcluded || key[i] == kTaken) && pos < a.budget) kept[pos++] = i;
  // total == n_tar + n_van by construction; the recent rows follow. The
  // guards only keep a broken count from writing outside this slab's row.
  for (int64_t j = threadIdx.x; j < a.rp; j += kSelectThreads)
    if (total + j < a.budget) kept[total + j] = static_cast<int32_t>(n_past + j);
}

__global__ void passthrough_kernel(int32_t* kept, int64_t n_slabs, int64_t n_tokens,
                                   int64_t budget) {
  const int64_t total = n_slabs * budget;
  for (int64_t g = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; g < total;
       g += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t j = g % budget;
    kept[g] = j < n_tokens ? static_cast<int32_t>(j) : -1;
  }
}

}  // namespace

size_t select_smem_bytes(int64_t n_tokens) {
  return (static_cast<size_t>((n_tokens + 3) & ~3LL) + kSelectBins) * sizeof(uint32_t);
}

cudaError_t select_prepare(int64_t max_tokens) {
  return cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(select_smem_bytes(max_tokens)));
}

cudaError_t launch_select(const SelectArgs& a, cudaStream_t st) {
  const size_t smem = select_smem_bytes(a.n_tokens - a.rp);
  select_kernel<<<static_cast<unsigned>(a.n_slabs), kSelectThreads, smem, st>>>(a);
  return cudaGetLastError();
}

cudaError_t launch_passthrough(int32_t* kept, int64_t n_slabs, int64_t n_tokens, int64_t budget,
                               cudaStream_t st) {
  const int64_t total = n_slabs * budget;
  const int64_t blocks = (total + 255) / 256;
  passthrough_kernel<<<static_cast<unsigned>(blocks < 4096 ? blocks : 4096), 256, 0, st>>>(
      kept, n_slabs, n_tokens, budget);
  return cudaGetLastError();
}

}  // namespace ipv
