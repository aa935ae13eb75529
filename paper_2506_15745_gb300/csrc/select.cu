// Step (iii) of the compression pass: the split-budget selection.
//
// Per (layer, KV head) slab (InfiniPot-V Sec. 3.3; Algorithm 1 steps 3-5):
// the r*p recent tokens are kept; the n_tar past tokens of highest s_TaR are
// taken; then the n_van past tokens of highest s_VaN among those TaR left
// (Algorithm 2 forces TaR picks to max(VaN) before its final TopK, which is
// the same as excluding them). Ties go to the lower token index. The kept
// set is written as ascending row indices.
//
// One 1024-thread CTA per slab; the scores are turned into order-preserving
// uint32 keys held in shared memory. A top-k threshold is found by repeated
// histogramming: the current key window [lo, hi] is split into 2048 equal
// integer bins, the bin holding the k-th largest key becomes the next window
// (at most 3 rounds for 32-bit keys). Tokens above the threshold key are
// taken, and of the tokens equal to it the lowest-index ones, counted with a
// block-wide prefix sum in index order.
#include "ipv_common.cuh"

namespace ipv {
namespace {

constexpr uint32_t kTaken = 0xFFFFFFFFu;    // VaN pick (never a score key)
constexpr uint32_t kExcluded = 0u;          // TaR pick, excluded from the VaN stage
constexpr uint32_t kNoBin = 0xFFFFFFFFu;

struct BlockShared {
  uint32_t warp_a[32];
  uint32_t warp_b[32];
  uint32_t bcast[8];
};

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

// Block-wide min and max of candidate keys (key >= 1); broadcast to all.
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

// Threshold of the k largest candidate keys (candidates: key >= 1) among
// key[0..n). The k winners are: every candidate with key > *T, plus the
// *take_eq lowest-index candidates with key == *T. *cnt_eq is the number of
// candidates with key == *T (only meaningful when *take_eq > 0).
// Requires 1 <= k <= number of candidates (n_cand).
__device__ void find_threshold(const uint32_t* key, int n, uint32_t k, uint32_t n_cand,
                               uint32_t* hist, BlockShared& sh, uint32_t* T, uint32_t* take_eq,
                               uint32_t* cnt_eq) {
  if (k >= n_cand) {  // every candidate is taken
    *T = 0u;
    *take_eq = 0u;
    *cnt_eq = 0u;
    return;
  }
  uint32_t lo = 0xFFFFFFFFu, hi = 0u;
  for (int i = threadIdx.x; i < n; i += kSelectThreads) {
    const uint32_t x = key[i];
    if (x >= 1u) {
      lo = min(lo, x);
      hi = max(hi, x);
    }
  }
  block_minmax(lo, hi, &lo, &hi, sh);
  uint32_t k_rem = k, cnt = n_cand;
  // The window shrinks at least 2048-fold per round, so 32-bit keys converge
  // in 4 rounds; the hard limit only guards against a broken invariant.
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
    // Thread t owns bins 2047-2t and 2046-2t (descending); an exclusive scan
    // gives the count of candidates in the bins above them.
    const int ba = kSelectBins - 1 - 2 * threadIdx.x, bb = ba - 1;
    const uint32_t ha = hist[ba], hb = hist[bb];
    if (threadIdx.x == 0) sh.bcast[2] = kNoBin;  // published by the scan's barriers
    uint32_t tot;
    const uint32_t above_a = block_excl_scan(ha + hb, &tot, sh);
    const uint32_t above_b = above_a + ha;
    if (above_a < k_rem && k_rem <= above_a + ha) {
      sh.bcast[2] = ba;
      sh.bcast[3] = above_a;
      sh.bcast[4] = ha;
    } else if (above_b < k_rem && k_rem <= above_b + hb) {
      sh.bcast[2] = bb;
      sh.bcast[3] = above_b;
      sh.bcast[4] = hb;
    }
    __syncthreads();
    const uint32_t bsel = sh.bcast[2], above = sh.bcast[3], cnt_b = sh.bcast[4];
    __syncthreads();
    if (bsel == kNoBin) break;  // fewer candidates than k_rem: cannot happen
    k_rem -= above;
    // Keys x with floor((x-lo)*2048/W) == bsel form [lo + ceil(bsel W/2048), lo + ceil((bsel+1) W/2048) - 1].
    const uint32_t lo_b = lo + static_cast<uint32_t>((bsel * W + kSelectBins - 1) / kSelectBins);
    const uint32_t hi_b =
        lo + static_cast<uint32_t>(((bsel + 1) * W + kSelectBins - 1) / kSelectBins) - 1u;
    if (cnt_b == k_rem) {  // the whole bin is taken: threshold just below it
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
  *take_eq = k_rem;
  *cnt_eq = cnt;
}

// Rank-among-ties bookkeeping: each thread walks the contiguous chunk
// [c0, c1) of indices; returns the number of candidates equal to T in the
// chunks of lower-numbered threads.
__device__ uint32_t ties_before(const uint32_t* key, int c0, int c1, uint32_t T, BlockShared& sh) {
  uint32_t mine = 0u;
  for (int i = c0; i < c1; ++i) mine += (key[i] == T) ? 1u : 0u;
  uint32_t tot;
  return block_excl_scan(mine, &tot, sh);
}

__global__ void __launch_bounds__(kSelectThreads, 1) select_kernel(SelectArgs a) {
  extern __shared__ uint32_t sm_key[];
  __shared__ BlockShared sh;
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
  for (int i = threadIdx.x; i < n_past; i += kSelectThreads) key[i] = score_key(tar[i]);
  __syncthreads();
  uint32_t T = 0xFFFFFFFFu, take = 0u, cnt_eq = 0u;  // default: nothing taken
  if (a.n_tar > 0)
    find_threshold(key, n_past, static_cast<uint32_t>(a.n_tar), static_cast<uint32_t>(n_past),
                   hist, sh, &T, &take, &cnt_eq);
  uint32_t rank = (take > 0u && take < cnt_eq) ? ties_before(key, c0, c1, T, sh) : 0u;
  const bool all_ties = take >= cnt_eq;
  for (int i = c0; i < c1; ++i) {
    const uint32_t x = key[i];
    bool pick = x > T && a.n_tar > 0;
    if (x == T && take > 0u) pick = all_ties || (rank++ < take);
    key[i] = pick ? kExcluded : score_key(van[i]);
  }
  __syncthreads();

  // VaN stage over the past tokens TaR left (keys >= 1).
  const uint32_t n_rest = static_cast<uint32_t>(n_past - a.n_tar);
  T = 0xFFFFFFFFu;
  take = 0u;
  cnt_eq = 0u;
  if (a.n_van > 0)
    find_threshold(key, n_past, static_cast<uint32_t>(a.n_van), n_rest, hist, sh, &T, &take,
                   &cnt_eq);
  rank = (take > 0u && take < cnt_eq) ? ties_before(key, c0, c1, T, sh) : 0u;
  const bool all_ties_v = take >= cnt_eq;
  for (int i = c0; i < c1; ++i) {
    const uint32_t x = key[i];
    if (x == kExcluded) continue;
    bool pick = x > T && a.n_van > 0;
    if (x == T && take > 0u) pick = all_ties_v || (rank++ < take);
    if (pick) key[i] = kTaken;
  }
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
