// Layer-adaptive pooling of VaN, used by the VaN stage when the library is
// set up with van_pool (InfiniPot-V Sec. 3.2 "Layer-wise Adaptive Pooling";
// Algorithm 2: CV = sigma / mu of the layer's VaN, pool size g(CV), then an
// average pool of every frame's VaN map).
//
// One 1024-thread block per (layer, KV head) slab, in two phases:
//  1. CV of the slab's layer over all its heads and cached rows, in fp32 with
//     a fixed reduction order (one sweep of sums shifted by the layer's first
//     value), so every block of a layer reaches the same bits and the same
//     pool size k.
//  2. For k > 1, each warp takes whole frames: round-robin for a cache that
//     was never compacted, else the frames that start in the 64-row chunks
//     it claims (pool_staged). A whole frame's (VaN, 1) pairs are scattered
//     into a dense grid_h x grid_w map in shared memory ((0, 0) where no
//     token is cached). Window sums and counts are separable: along the grid
//     row for every cell, then along the column; their quotient is the mean.
//     Sums are direct (k terms each), never running sums, so a large value
//     leaving the window cannot leave rounding behind. For k = 1 the rows
//     are copied.
// Frames: rows carry (frame id, patch id) in increasing order, or derive
// them as (n div p, n mod p) for a cache that was never compacted; a frame is
// a maximal run of rows with one frame id.
//
// The work is small (VaN is 4 bytes per token, read from L2 where the
// scoring kernel just wrote it); the block count is the slab count.
#include <cmath>

#include "ipv_common.cuh"

namespace ipv {
namespace {

constexpr size_t kPoolSmem = 200 * 1024;



// Block-wide sum of pairs in a fixed order: a butterfly within each warp
// (every lane ends with the same bits), then warp 0 over the per-warp totals.
__device__ float2 block_sum2(float2 x, float2* red) {
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) {
    x.x += __shfl_xor_sync(0xffffffffu, x.x, off);
    x.y += __shfl_xor_sync(0xffffffffu, x.y, off);
  }
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (lane == 0) red[warp] = x;
  __syncthreads();
  if (warp == 0) {
    float2 t = lane < static_cast<int>(blockDim.x >> 5) ? red[lane] : make_float2(0.0f, 0.0f);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) {
      t.x += __shfl_xor_sync(0xffffffffu, t.x, off);
      t.y += __shfl_xor_sync(0xffffffffu, t.y, off);
    }
    if (lane == 0) red[32] = t;
  }
  __syncthreads();
  return red[32];
}

// This thread's share of sum(x - c) and sum((x - c)^2) over the layer's count
// values (elements threadIdx.x + i * blockDim.x), ten 16-byte loads in
// flight (a layer of 4 x 9408 values in one round), fixed order. The shift c (the layer's first value) keeps the
// one-sweep variance E[(x - c)^2] - E[x - c]^2 free of cancellation.
__device__ float2 layer_sums4(const float* lv, int64_t count, float c) {
  const float4* lv4 = reinterpret_cast<const float4*>(lv);
  const int n4 = static_cast<int>(count / 4), step = blockDim.x;
  constexpr int kU = 10;
  float2 a[4] = {};
  for (int i0 = threadIdx.x; i0 < n4; i0 += kU * step) {
    float4 x[kU];
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const int i = i0 + u * step;
      x[u] = i < n4 ? lv4[i] : make_float4(c, c, c, c);  // c contributes 0
    }
#pragma unroll
    for (int u = 0; u < kU; ++u) {
      const float d0 = x[u].x - c, d1 = x[u].y - c, d2 = x[u].z - c, d3 = x[u].w - c;
      a[u & 3].x += (d0 + d1) + (d2 + d3);
      a[u & 3].y += (d0 * d0 + d1 * d1) + (d2 * d2 + d3 * d3);
    }
  }
  return make_float2((a[0].x + a[1].x) + (a[2].x + a[3].x), (a[0].y + a[1].y) + (a[2].y + a[3].y));
}

__device__ float2 layer_sums1(const float* lv, int64_t count, float c) {
  float2 acc = make_float2(0.0f, 0.0f);
  for (int64_t i = threadIdx.x; i < count; i += blockDim.x) {
    const float d = lv[i] - c;
    acc.x += d;
    acc.y += d * d;
  }
  return acc;
}

// Row indices fit in 32 bits (n_tokens <= IPV_MAX_TOKENS).
struct RowIds {
  const uint16_t* pid;  // this slab's ids, or nullptr
  const uint32_t* fid;
  int p;
};

// Pools the whole frame of rows [a, b) of a never-compacted cache (row a + q
// is patch q; a whole warp) with window radius HALF, separably. cell: this
// warp's p float2 (VaN, 1) of cached positions, (0, 0) elsewhere; row: p
// float2 window sums along grid rows; ij: the block's (i, j) of every cell.
// Cells are contiguous in c, so a warp's accesses are conflict-free; the
// window sums are unrolled (2 HALF + 1 predicated loads in flight).
template <int HALF>
__device__ void pool_frame(const PoolArgs& pa, const RowIds& ids, const float* sv, float* out,
                           int a, int b, float2* cell, float2* row, const short2* ij) {
  const int lane = threadIdx.x & 31;
  const int p = ids.p, gw = pa.grid_w, gh = pa.grid_h;
  for (int c = lane; c < p; c += 32) cell[c] = make_float2(0.0f, 0.0f);
  __syncwarp();
#pragma unroll 4
  for (int m = a + lane; m < b; m += 32) {  // independent loads, several in flight
    cell[m - a] = make_float2(sv[m], 1.0f);
  }
  __syncwarp();
  for (int c = lane; c < p; c += 32) {  // sums and counts along the grid row
    const short2 t = ij[c];
    float2 x[2 * HALF + 1];
#pragma unroll
    for (int d = -HALF; d <= HALF; ++d) {
      const int jj = t.y + d;
      x[d + HALF] = (jj >= 0 && jj < gw) ? cell[c + d] : make_float2(0.0f, 0.0f);
    }
    float2 acc = x[0];
#pragma unroll
    for (int u = 1; u <= 2 * HALF; ++u) {
      acc.x += x[u].x;
      acc.y += x[u].y;
    }
    row[c] = acc;
  }
  __syncwarp();
  for (int c = lane; c < p; c += 32) {  // then along the grid column: the window mean
    const short2 t = ij[c];
    float2 x[2 * HALF + 1];
#pragma unroll
    for (int d = -HALF; d <= HALF; ++d) {
      const int ii = t.x + d;
      x[d + HALF] = (ii >= 0 && ii < gh) ? row[c + d * gw] : make_float2(0.0f, 0.0f);
    }
    float2 acc = x[0];
#pragma unroll
    for (int u = 1; u <= 2 * HALF; ++u) {
      acc.x += x[u].x;
      acc.y += x[u].y;
    }
    cell[c].x = __fdividef(acc.x, acc.y);  // cells without a cached token are never read
  }
  __syncwarp();
  for (int m = a + lane; m < b; m += 32) out[m] = cell[m - a].x;
  __syncwarp();  // the arrays are reused by this warp's next frame
}

// ---------------------------------------------------------------- layout
// Dynamic shared memory of the pooling block:
//   nw per-warp maps of max(4 p, 2 (gh + 2 kPad)(gw + 2 kPad)) floats: the two
//     p-float2 arrays of pool_frame (whole frames) or the zero-padded
//     (VaN, 1) map of pool_tokens (caches with ids);
//   the p-entry (i, j) table;
//   the row staging of caches with ids: VaN and frame id (4 bytes each) and
//     patch id (2 bytes) of stage_rows rows.
constexpr int kPad = 3;  // radius of the largest pool (k = 7)

struct PoolLayout {
  int nw;          // warps that pool (0: the frame does not fit)
  int map_floats;  // per warp
  int stage_rows;  // rows staged at once
  int tile;        // rows whose frames one staging covers (stage_rows - p - 1)
};

__host__ __device__ inline PoolLayout pool_layout(int gh, int gw) {
  PoolLayout L{};
  const int p = gh * gw;
  const int padded = 2 * (gh + 2 * kPad) * (gw + 2 * kPad);
  L.map_floats = 4 * p > padded ? 4 * p : padded;
  const size_t map_bytes = static_cast<size_t>(L.map_floats) * sizeof(float);
  int nw = static_cast<int>((kPoolSmem * 11 / 20) / map_bytes);  // maps take at most 55%
  nw = nw < 32 ? nw : 32;
  if (nw < 1) return PoolLayout{};
  const size_t rest = kPoolSmem - nw * map_bytes - static_cast<size_t>(p) * 4;
  L.stage_rows = static_cast<int>(rest / 10) & ~3;
  L.tile = L.stage_rows - p - 1;
  if (L.tile < 32) return PoolLayout{};
  L.nw = nw;
  return L;
}

// Pools every cached token of the frame rows [a, b) (a whole warp): the mean
// of the (VaN, 1) pairs in its (2 HALF + 1)^2 window of the zero-padded map.
// The map is zero on entry and on exit. Rows come from the block's staging:
// stage index m - st0. Two ways, whichever takes fewer shared-memory reads:
//  - direct: every token sums its whole window, (2 HALF + 1)^2 reads each;
//  - separable (p <= 32 kSepCells): each lane sums its interior cells along
//    the grid row into registers, writes those row sums back over the map's
//    interior, and every token then sums its column of row sums; padding
//    rows and columns stay zero. All interior cells are cleared afterwards.
constexpr int kSepCells = 8;  // interior cells per lane of the separable way

template <int HALF>
__device__ void pool_tokens(const PoolArgs& pa, int p, const float* s_van, const uint16_t* s_pid,
                            int st0, float* out, int a, int b, float2* map, const short2* ij) {
  constexpr int W = 2 * HALF + 1;
  const int lane = threadIdx.x & 31;
  const int cp = pa.grid_w + 2 * kPad;
  for (int m = a + lane; m < b; m += 32) {
    const int q = s_pid[m - st0];
    if (q < p) {
      const short2 t = ij[q];
      map[(t.x + kPad) * cp + t.y + kPad] = make_float2(s_van[m - st0], 1.0f);
    }
  }
  __syncwarp();
  const int n = b - a;
  const bool sep = p <= 32 * kSepCells && p * W + n * W + 2 * p < n * W * W;  // warp-uniform
  if (sep) {
    float2 rs[kSepCells];
#pragma unroll
    for (int u = 0; u < kSepCells; ++u) {
      const int c = lane + 32 * u;
      rs[u] = make_float2(0.0f, 0.0f);
      if (c < p) {
        const short2 t = ij[c];
        const float2* r = map + (t.x + kPad) * cp + t.y + kPad;
        float2 x[W];
#pragma unroll
        for (int dj = -HALF; dj <= HALF; ++dj) x[dj + HALF] = r[dj];
#pragma unroll
        for (int d = 0; d < W; ++d) {
          rs[u].x += x[d].x;
          rs[u].y += x[d].y;
        }
      }
    }
    __syncwarp();  // every row sum is read before any is written back
#pragma unroll
    for (int u = 0; u < kSepCells; ++u) {
      const int c = lane + 32 * u;
      if (c < p) {
        const short2 t = ij[c];
        map[(t.x + kPad) * cp + t.y + kPad] = rs[u];
      }
    }
    __syncwarp();
  }
  for (int m = a + lane; m < b; m += 32) {
    const int q = s_pid[m - st0];
    float y = __int_as_float(0x7fc00000);  // NaN: no grid position
    if (q < p) {
      const short2 t = ij[q];
      const float2* c = map + (t.x + kPad) * cp + t.y + kPad;
      float2 acc = make_float2(0.0f, 0.0f);
      if (sep) {
        float2 x[W];
#pragma unroll
        for (int di = -HALF; di <= HALF; ++di) x[di + HALF] = c[di * cp];
#pragma unroll
        for (int d = 0; d < W; ++d) {
          acc.x += x[d].x;
          acc.y += x[d].y;
        }
      } else {
#pragma unroll
        for (int di = -HALF; di <= HALF; ++di) {
          const float2* r = c + di * cp;
          float2 x[W];
#pragma unroll
          for (int dj = -HALF; dj <= HALF; ++dj) x[dj + HALF] = r[dj];
#pragma unroll
          for (int u = 0; u < W; ++u) {
            acc.x += x[u].x;
            acc.y += x[u].y;
          }
        }
      }
      y = __fdividef(acc.x, acc.y);
    }
    out[m] = y;
  }
  __syncwarp();
  if (sep) {
    for (int c = lane; c < p; c += 32) {
      const short2 t = ij[c];
      map[(t.x + kPad) * cp + t.y + kPad] = make_float2(0.0f, 0.0f);
    }
  } else {
    for (int m = a + lane; m < b; m += 32) {
      const int q = s_pid[m - st0];
      if (q < p) {
        const short2 t = ij[q];
        map[(t.x + kPad) * cp + t.y + kPad] = make_float2(0.0f, 0.0f);
      }
    }
  }
  __syncwarp();
}

// Phase 2 of a slab with patch and frame ids (a compacted cache): the rows
// are staged tile by tile in shared memory; a frame (a maximal run of one
// frame id) is pooled by the warp that claims the chunk of kPoolChunk rows
// holding its first row. Frames are at most p rows long when rows are in
// (frame, patch) order, so a tile's frames end inside its staging. Such
// caches hold many small frames (the survivors of earlier passes): a warp
// takes 32 rows at a time, from a frame start, and pools every frame that
// ends among them pairwise over shuffles (same frame, within HALF rows and
// columns); a frame of more than 32 rows goes through the map (pool_tokens).
// Chunks are claimed from a shared counter, the last rows first: the newest
// frames, the largest and costliest, go out before the many small ones that
// fill in behind them, so the warps finish together.
constexpr int kPoolChunk = 64;

template <int HALF>
__device__ void pool_staged(const PoolArgs& pa, const RowIds& ids, const float* sv, float* out,
                            int n_rows, const PoolLayout& L, float* maps, const short2* ij,
                            float* s_van, uint32_t* s_fid, uint16_t* s_pid) {
  __shared__ int s_claim;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int p = ids.p;
  float2* map = reinterpret_cast<float2*>(maps + static_cast<size_t>(warp) * L.map_floats);
  for (int t0 = 0; t0 < n_rows; t0 += L.tile) {  // block-uniform
    const int t1 = min(n_rows, t0 + L.tile);
    const int st0 = max(0, t0 - 1);                // one row before the tile: start detection
    const int e1 = min(n_rows, t1 + p);            // the tile's last frame ends before e1
    __syncthreads();                               // the previous tile's staging and claims are done
    if (threadIdx.x == 0) s_claim = 0;
    if (t0 == 0) {
      // The first tile's ids were staged before the wait for the scores and
      // its VaN while the CV was summed.
      cp_async_wait_all();
    } else {
#pragma unroll 4
      for (int m = st0 + threadIdx.x; m < e1; m += blockDim.x) {
        s_van[m - st0] = sv[m];
        s_fid[m - st0] = ids.fid[m];
        s_pid[m - st0] = ids.pid[m];
      }
    }
    __syncthreads();
    if (warp >= L.nw) continue;
    const int n_chunks = (t1 - t0 + kPoolChunk - 1) / kPoolChunk;
    for (;;) {  // warp-uniform
      int c = 0;
      if (lane == 0) c = atomicAdd(&s_claim, 1);
      c = __shfl_sync(0xffffffffu, c, 0);
      if (c >= n_chunks) break;
      const int lo = t0 + (n_chunks - 1 - c) * kPoolChunk;
      const int hi = min(t1, lo + kPoolChunk);
      // The first frame start at or after lo.
      int a = hi;
      for (int base = lo; base < hi; base += 32) {  // warp-uniform
        const int n = base + lane;
        const bool st = n < hi && (n == 0 || s_fid[n - st0] != s_fid[n - 1 - st0]);
        const unsigned mask = __ballot_sync(0xffffffffu, st);
        if (mask) {
          a = base + __ffs(mask) - 1;
          break;
        }
      }
      while (a < hi) {  // warp-uniform; a is a frame start
        // Rows [a, a + 32), one per lane: pool every frame that ends among them.
        const int m = a + lane;
        const bool valid = m < e1;
        const uint32_t f = valid ? s_fid[m - st0] : 0u;
        const bool st = valid && (lane == 0 || f != s_fid[m - 1 - st0]);
        const unsigned starts = __ballot_sync(0xffffffffu, st);
        const unsigned foreign = __ballot_sync(0xffffffffu, st && m >= hi);  // other warps' frames
        int end;
        if (foreign) {
          end = __ffs(foreign) - 1;
        } else {
          const int nx = a + 32;
          const bool next_starts = nx >= e1 || s_fid[nx - st0] != s_fid[nx - 1 - st0];
          end = next_starts ? 32 : 31 - __clz(starts);  // leave a frame cut at a + 32 to the next batch
        }
        end = min(end, e1 - a);  // rows past the staging are not read
        if (end == 0) {  // one frame of more than 32 rows starts at a
          int b = e1;
          for (int c = a + 1; c < e1; c += 32) {  // end of the run, inside the staging
            const int mm = c + lane;
            const unsigned other = __ballot_sync(0xffffffffu, mm < e1 && s_fid[mm - st0] != s_fid[a - st0]);
            if (other) {
              b = c + __ffs(other) - 1;
              break;
            }
          }
          pool_tokens<HALF>(pa, p, s_van, s_pid, st0, out, a, b, map, ij);
          a = b;
          continue;
        }
        // Pairwise: each lane reads the tokens of its own frame (lanes fs..fe-1
        // of the batch) in row order; one counts when it lies within HALF grid
        // rows and columns. The loop runs as long as the batch's longest frame.
        // A token's grid row is offset by its frame's rank in the batch times
        // grid_h + HALF + 1, so tokens of other frames are never within HALF
        // rows and the loop needs no frame test; tokens without a position sit
        // at row 0xffff, columns 8 apart. Rows stay below 2^16: grid_h <= 2005
        // for a poolable grid, so 32 grid_h + 123 <= 64283.
        const bool mine = lane < end;
        const int q = mine ? s_pid[m - st0] : p;
        const float x = mine ? s_van[m - st0] : 0.0f;
        const bool has_pos = q < p;
        const unsigned in_batch = starts & (end == 32 ? 0xffffffffu : ((1u << end) - 1u));
        const unsigned upto = lane == 31 ? 0xffffffffu : ((2u << lane) - 1u);  // bits 0..lane
        const int fs = 31 - __clz(in_batch & upto);                           // my frame's first lane
        const unsigned after = in_batch & ~upto;
        const int fe = after ? __ffs(after) - 1 : end;                         // one past its last lane
        const int len = mine ? fe - fs : 0;
        const int max_len = static_cast<int>(__reduce_max_sync(0xffffffffu, static_cast<unsigned>(len)));
        const short2 t = has_pos ? ij[q] : make_short2(0, 0);
        const int rank = __popc(in_batch & upto) - 1;
        const int ti = has_pos ? t.x + rank * (pa.grid_h + HALF + 1) : 0xffff;
        const int tj = has_pos ? t.y : lane * 8;
        const uint32_t tij = (static_cast<uint32_t>(ti) << 16) | static_cast<uint32_t>(tj);
        float sum = 0.0f, cnt = 0.0f;
        for (int v = 0; v < max_len; ++v) {  // warp-uniform
          // Lanes past fe, or wrapped below fs, hold other frames.
          const int src = (fs + v) & 31;
          const uint32_t tu = __shfl_sync(0xffffffffu, tij, src);
          const float xu = __shfl_sync(0xffffffffu, x, src);
          const unsigned du = static_cast<unsigned>(static_cast<int>(tu >> 16) - ti + HALF);
          const unsigned dv = static_cast<unsigned>(static_cast<int>(tu & 0xffffu) - tj + HALF);
          if (du <= 2u * HALF && dv <= 2u * HALF) {
            sum += xu;
            cnt += 1.0f;
          }
        }
        if (mine) out[m] = has_pos ? __fdividef(sum, cnt) : __int_as_float(0x7fc00000);
        a += end;
      }
    }
  }
}

__global__ void __launch_bounds__(kPoolThreads, 1) pool_kernel(PoolArgs pa) {
  extern __shared__ float sm_pool[];
  __shared__ float2 red[33];
  pdl_trigger();
  const int64_t s = blockIdx.x;
  const int64_t layer = s / pa.n_heads;

  // What does not read the scores is set up before waiting for them: blocks
  // that start on SMs the scoring kernel has already left do it meanwhile.
  const int p = pa.grid_h * pa.grid_w;
  const PoolLayout L = pool_layout(pa.grid_h, pa.grid_w);
  float* maps = sm_pool;
  short2* ij = reinterpret_cast<short2*>(maps + static_cast<size_t>(L.nw) * L.map_floats);
  for (int c = threadIdx.x; c < p; c += blockDim.x)
    ij[c] = make_short2(static_cast<short>(c / pa.grid_w), static_cast<short>(c % pa.grid_w));
  RowIds ids;
  ids.pid = pa.patch_id ? pa.patch_id + s * pa.id_stride : nullptr;
  ids.fid = pa.frame_id ? pa.frame_id + s * pa.id_stride : nullptr;
  ids.p = p;
  const int n_rows = static_cast<int>(pa.n_rows);
  float* s_van = reinterpret_cast<float*>(ij + p);
  uint32_t* s_fid = reinterpret_cast<uint32_t*>(s_van + L.stage_rows);
  uint16_t* s_pid = reinterpret_cast<uint16_t*>(s_fid + L.stage_rows);
  if (ids.fid) {  // the zeroed maps and the first tile's ids (pool_staged's staging)
    for (int i = threadIdx.x; i < L.nw * L.map_floats; i += blockDim.x) maps[i] = 0.0f;
    const int e1 = min(n_rows, L.tile + p);
#pragma unroll 4
    for (int m = threadIdx.x; m < e1; m += blockDim.x) {
      s_fid[m] = ids.fid[m];
      s_pid[m] = ids.pid[m];
    }
  }
  pdl_wait();  // VaN comes from the scoring kernels
  const float* sv = pa.van + s * pa.n_tokens;
  if (ids.fid) {  // the first tile's VaN (pool_staged) is copied while the CV is summed
    const int e1 = min(n_rows, L.tile + p);
    for (int m = threadIdx.x; m < e1; m += blockDim.x) cp_async4(s_van + m, sv + m);
  }

  // Phase 1: CV of the layer (Algorithm 2: mu, sigma, CV = sigma / mu).
  const int64_t count = static_cast<int64_t>(pa.n_heads) * pa.n_tokens;
  const float* lv = pa.van + layer * count;
  const bool vec = (reinterpret_cast<uintptr_t>(lv) & 15u) == 0 && (count & 3) == 0;
  const float n_f = static_cast<float>(count);
  const float shift = lv[0];
  const float2 t = block_sum2(vec ? layer_sums4(lv, count, shift) : layer_sums1(lv, count, shift), red);
  const float dm = t.x / n_f;                   // mean - shift
  const float var = fmaxf(t.y / n_f - dm * dm, 0.0f);
  const float cv = sqrtf(var) / (shift + dm);
  // g(CV): 7, 5, 3, 1; a NaN CV passes no comparison and gets 1.
  const int k = cv < pa.tau[0] ? 7 : cv < pa.tau[1] ? 5 : cv < pa.tau[2] ? 3 : 1;
  if (pa.pool_size && s % pa.n_heads == 0 && threadIdx.x == 0) pa.pool_size[layer] = k;

  // Phase 2: the pooled VaN of rows [0, n_rows) of this slab.
  float* out = pa.pooled + s * pa.n_tokens;
  if (k == 1) {
    cp_async_wait_all();  // no copy into shared memory outlives the block
    for (int64_t n = threadIdx.x; n < pa.n_rows; n += blockDim.x) out[n] = sv[n];
    return;
  }
  const int warp = threadIdx.x >> 5;
  if (!ids.fid) {  // never compacted: whole p-row frames, dealt round-robin
    if (warp >= L.nw) return;  // block_sum2's barriers published the (i, j) table
    float2* cell = reinterpret_cast<float2*>(maps + static_cast<size_t>(warp) * L.map_floats);
    float2* row = cell + p;
    for (int a = warp * p; a < n_rows; a += L.nw * p) {
      const int b = min(n_rows, a + p);
      if (k == 7) pool_frame<3>(pa, ids, sv, out, a, b, cell, row, ij);
      else if (k == 5) pool_frame<2>(pa, ids, sv, out, a, b, cell, row, ij);
      else pool_frame<1>(pa, ids, sv, out, a, b, cell, row, ij);
    }
    return;
  }
  if (k == 7) pool_staged<3>(pa, ids, sv, out, n_rows, L, maps, ij, s_van, s_fid, s_pid);
  else if (k == 5) pool_staged<2>(pa, ids, sv, out, n_rows, L, maps, ij, s_van, s_fid, s_pid);
  else pool_staged<1>(pa, ids, sv, out, n_rows, L, maps, ij, s_van, s_fid, s_pid);
}

// Frame-level TaR (the "TaR Frame" ablation): every past row of unit
// blockIdx.x takes the mean of its frame's past-row scores. The rows of a
// tile are staged in shared memory (score, frame id); each warp takes the
// frames that start in its share, sums a frame lane by lane in row order then
// across lanes (fixed order), and writes the mean to all its rows.
constexpr int kMeanTile = 8192;

__global__ void __launch_bounds__(1024, 1) frame_mean_kernel(FrameMeanArgs a) {
  extern __shared__ float sm_fm[];
  pdl_trigger();
  pdl_wait();  // the scores come from the scoring kernels
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31, nw = blockDim.x >> 5;
  float* t = a.tar + blockIdx.x * a.n_tokens;
  const uint32_t* fid = a.frame_id ? a.frame_id + blockIdx.x * a.id_stride : nullptr;
  const int n_past = static_cast<int>(a.n_past), p = a.p;
  float* s_val = sm_fm;
  uint32_t* s_fid = reinterpret_cast<uint32_t*>(sm_fm + kMeanTile + p + 1);
  for (int t0 = 0; t0 < n_past; t0 += kMeanTile) {  // block-uniform
    const int t1 = min(n_past, t0 + kMeanTile);
    const int st0 = max(0, t0 - 1);
    const int e1 = min(n_past, t1 + p);  // a frame is at most p rows
    __syncthreads();
    for (int m = st0 + threadIdx.x; m < e1; m += blockDim.x) {
      s_val[m - st0] = t[m];
      s_fid[m - st0] = fid ? fid[m] : static_cast<uint32_t>(m / p);
    }
    __syncthreads();
    const int share = (t1 - t0 + nw - 1) / nw;
    const int lo = t0 + warp * share, hi = min(t1, lo + share);
    for (int base = lo; base < hi; base += 32) {  // warp-uniform
      const int n = base + lane;
      const bool st = n < hi && (n == 0 || s_fid[n - st0] != s_fid[n - 1 - st0]);
      unsigned mask = __ballot_sync(0xffffffffu, st);
      while (mask) {
        const int f0 = base + __ffs(mask) - 1;
        mask &= mask - 1;
        const uint32_t f = s_fid[f0 - st0];
        int f1 = e1;
        for (int c = f0 + 1; c < e1; c += 32) {  // end of the run, inside the staging
          const int mm = c + lane;
          const unsigned other = __ballot_sync(0xffffffffu, mm < e1 && s_fid[mm - st0] != f);
          if (other) {
            f1 = c + __ffs(other) - 1;
            break;
          }
        }
        float sum = 0.0f;
        for (int m = f0 + lane; m < f1; m += 32) sum += s_val[m - st0];
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
        const float mean = sum / static_cast<float>(f1 - f0);
        for (int m = f0 + lane; m < f1; m += 32) t[m] = mean;
      }
    }
  }
}

}  // namespace

cudaError_t launch_frame_mean(const FrameMeanArgs& a, cudaStream_t st) {
  if (a.p > kMaxPoolFrame) return cudaErrorInvalidValue;
  const size_t smem = 2 * static_cast<size_t>(kMeanTile + a.p + 1) * sizeof(float);
  cudaError_t e = launch(frame_mean_kernel, static_cast<unsigned>(a.units), 1024, smem, st, true, a);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

size_t pool_smem_bytes(int gh, int gw, bool staged) {
  const PoolLayout L = pool_layout(gh, gw);
  if (L.nw == 0) return 0;
  // Without ids (a never-compacted cache) nothing is staged: a smaller
  // request lets the block start beside the scoring kernel's last blocks.
  return staged ? kPoolSmem
                : static_cast<size_t>(L.nw) * L.map_floats * sizeof(float) + static_cast<size_t>(gh) * gw * 4;
}

cudaError_t pool_prepare() {
  cudaError_t e = cudaFuncSetAttribute(pool_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(kPoolSmem));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(frame_mean_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(2 * (kMeanTile + kMaxPoolFrame + 1) * sizeof(float)));
}

cudaError_t launch_pool(const PoolArgs& a, cudaStream_t st, bool pdl) {
  const size_t smem = pool_smem_bytes(a.grid_h, a.grid_w, a.frame_id != nullptr);
  if (smem == 0) return cudaErrorInvalidValue;
  cudaError_t e = launch(pool_kernel, static_cast<unsigned>(a.n_slabs), kPoolThreads, smem, st, pdl, a);
  return e == cudaSuccess ? cudaGetLastError() : e;
}

}  // namespace ipv
