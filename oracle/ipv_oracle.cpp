// InfiniPot-V compression pass: plain CPU oracle (fp64, single-threaded).
//
// TEST INFRASTRUCTURE ONLY. Nothing on the product path may link, load or call
// this file. Its only users are tests/, __graft_entry__.smoke() and the
// cpu_baseline / reference legs of bench.py. It shares no code, header or
// constant with the CUDA path (paper_2506_15745_gb300/csrc); the two meet only
// on the bytes of the synthetic inputs.
//
// What it computes, per (layer, KV head) slab, following InfiniPot-V
// (arXiv 2506.15745):
//   * TaR score, Sec. 3.1 Eq. (tar): for a past token at frame t, patch (i,j),
//       s = -(1/r) * sum_{t'=1..r} cos(K_past[t,i,j], K_recent[t',i,j]),
//     with the cache viewed as f frames of p = |M|/f patches, the r latest
//     frames "recent" and the rest "past" (Sec. 3.1; Algorithm 2 reshape).
//     The sum of r cosines is evaluated literally, term by term.
//   * VaN score, Sec. 3.2: s = ||V[t,i,j]||_2.
//   * Selection, Algorithm 1 steps (3)-(5) with the Sec. 3.3 split: the r
//     recent frames are always kept and count inside the TaR share
//     (alpha*|C| - len(K_recent)); the TaR share is the top of s_TaR over the
//     past tokens; the rest of |C| is filled by the top of s_VaN over the past
//     tokens TaR did not take (Algorithm 2 forces TaR picks to max(VaN) before
//     its final TopK, which is the same as excluding them). Ties go to the
//     lower token index; NaN scores rank below every number.
//   * Compaction, Sec. 3.1 / Algorithm 2 last step: K~ = K[:, J, :], the kept
//     rows copied in ascending index order.
//
// Readings where the paper is silent (each is listed in the design notes):
// alpha*|C| is floored; r defaults to max(1, floor(f/8 + 1/2)) (Appendix B.2
// standardises r = 0.125 f); a cache at or below |C| tokens is passed through
// (Algorithm 1 triggers only when len(K) >= |M| > |C|); cosine uses
// max(||x||, 1e-12) in each denominator so that a zero vector has cosine 0;
// past-token patch coordinates come from an optional per-token patch-id array
// (else n mod p), recent rows are whole frames at rows N - r p + t' p + q.
//
// Layer-adaptive VaN pooling (Sec. 3.2 "Layer-wise Adaptive Pooling";
// Algorithm 2), used when the pass is asked for it: per layer, the mean mu and
// standard deviation sigma of VaN over all heads and all cached tokens give
// CV = sigma / mu; g(CV) = 7, 5, 3, 1 for CV < tau_1, < tau_2, < tau_3, >= tau_3
// picks an average-pool size k; each token's pooled VaN is the mean VaN of the
// tokens of its own frame inside the k x k window centred on its grid position
// (stride 1). Readings: sigma is the population standard deviation; window
// positions outside the grid, or whose token is no longer cached, are left
// out of the mean (no zero padding); the VaN stage of the selection ranks the
// pooled values. Where rows carry patch ids they also carry frame ids (the
// frame each token came from); a never-compacted cache has frame n div p.
//
// Per-layer shared index set (Sec. 3.1: K is H x N x D and the compressed
// cache is K[:, I, :], one index set I for all H heads of a layer; likewise
// Algorithm 2's I_l and J_l per layer), used when the pass is asked for it:
// a token's key and value are its H x D blocks, the cosine of Eq. (tar) is
// the l2-normalised (Frobenius) cosine of the concatenated H*D vectors, and
// VaN is their Frobenius norm. Selection then runs once per layer and every
// head of the layer is compacted with that layer's indices.
//
// Ablation variants (Sec. 4 ablation study, "TaR Reverse", "VaN Reverse",
// "TaR Frame", "Uniform Select"), used when the pass is asked for one: a
// reversed stage keeps the lowest scores instead of the highest (its scores
// negated; NaN still ranks last, ties still go to the lower index); the
// frame-level TaR gives each past token the mean TaR of the cached past
// tokens of its frame; Uniform Select (Sec. 4, KV cache compression details:
// frames at regular intervals, all their tokens kept) ignores the scores and
// keeps k = |C|/p whole frames of the F = |M|/p frames of the frame view,
// every (F/k)-th frame counting back from the newest: frames
// F - 1 - floor(i F / k), i = 0..k-1.
//
// Element types: bf16 (widened exactly: bits << 16) or fp32, widened to double.

#include <algorithm>
#include <cmath>
#include <cstdint>
#include <cstring>
#include <limits>
#include <map>
#include <vector>

namespace {

double widen(const void* base, int is_bf16, int64_t idx) {
  if (is_bf16) {
    uint16_t h = static_cast<const uint16_t*>(base)[idx];
    uint32_t u = static_cast<uint32_t>(h) << 16;
    float f;
    std::memcpy(&f, &u, sizeof f);
    return static_cast<double>(f);
  }
  return static_cast<double>(static_cast<const float*>(base)[idx]);
}

// Row n of slab s of a [n_slabs][cap][D] tensor, widened to double.
void load_row(const void* base, int is_bf16, int64_t s, int64_t cap, int D,
              int64_t n, std::vector<double>& out) {
  out.resize(D);
  const int64_t off = (s * cap + n) * static_cast<int64_t>(D);
  for (int d = 0; d < D; ++d) out[d] = widen(base, is_bf16, off + d);
}

double dot(const std::vector<double>& a, const std::vector<double>& b) {
  double acc = 0.0;
  for (size_t d = 0; d < a.size(); ++d) acc += a[d] * b[d];
  return acc;
}

double l2norm(const std::vector<double>& a) { return std::sqrt(dot(a, a)); }

// cos(a, b) = a.b / (max(|a|,eps) max(|b|,eps)); a zero vector gives 0.
double cosine(const std::vector<double>& a, const std::vector<double>& b) {
  const double eps = 1e-12;
  return dot(a, b) / (std::max(l2norm(a), eps) * std::max(l2norm(b), eps));
}

// Strict "x ranks above y" for (score desc, index asc), NaN lowest.
bool ranks_above(double xs, int64_t xi, double ys, int64_t yi) {
  const bool xn = std::isnan(xs), yn = std::isnan(ys);
  if (xn || yn) {
    if (xn && yn) return xi < yi;
    return yn;  // a number ranks above NaN
  }
  if (xs != ys) return xs > ys;
  return xi < yi;
}

}  // namespace

extern "C" {

// Recent-frame count r. Appendix B.2 fixes r = 0.125 f as the default ratio;
// rounding to an integer frame count is our reading (half rounds up), never
// below one frame. A positive override is returned unchanged.
int oracle_recent_frames(int64_t n_frames, int override_r) {
  if (override_r > 0) return override_r;
  const int64_t r = static_cast<int64_t>(std::floor(n_frames / 8.0 + 0.5));
  return static_cast<int>(std::max<int64_t>(1, r));
}

// TaR and VaN scores for every past token of every slab (Sec. 3.1 Eq. tar,
// Sec. 3.2). k, v: [n_slabs][cap][D]; patch_id: [n_slabs][cap] or NULL.
// tar_out, van_out: [n_slabs][n_tokens]; entries of the r recent frames are
// written as 0 (those tokens are always kept and are never scored).
// Returns 0, or -1 on bad arguments (incl. a patch id >= p).
int oracle_scores(const void* k, const void* v, int is_bf16, int64_t n_slabs,
                  int64_t cap, int D, int64_t n_tokens, int p, int r,
                  const uint16_t* patch_id, double* tar_out, double* van_out) {
  if (!k || !v || !tar_out || !van_out || n_slabs < 0 || D <= 0 || p <= 0 ||
      r <= 0 || n_tokens < 0 || n_tokens > cap || n_tokens % p != 0)
    return -1;
  const int64_t rp = static_cast<int64_t>(r) * p;
  if (rp > n_tokens) return -1;
  const int64_t n_past = n_tokens - rp;
  std::vector<double> kp, kr, vv;
  for (int64_t s = 0; s < n_slabs; ++s) {
    double* tar = tar_out + s * n_tokens;
    double* van = van_out + s * n_tokens;
    for (int64_t n = 0; n < n_tokens; ++n) tar[n] = van[n] = 0.0;
    for (int64_t n = 0; n < n_past; ++n) {
      const int64_t q = patch_id ? patch_id[s * cap + n] : n % p;
      if (q < 0 || q >= p) return -1;
      load_row(k, is_bf16, s, cap, D, n, kp);
      double sum_cos = 0.0;
      for (int t = 0; t < r; ++t) {
        load_row(k, is_bf16, s, cap, D, n_past + static_cast<int64_t>(t) * p + q, kr);
        sum_cos += cosine(kp, kr);
      }
      tar[n] = -sum_cos / r;
      load_row(v, is_bf16, s, cap, D, n, vv);
      van[n] = l2norm(vv);
    }
  }
  return 0;
}

// The H head-rows of token n of layer l, concatenated: slabs l*H .. l*H+H-1.
static void load_token(const void* base, int is_bf16, int64_t l, int H, int64_t cap, int D, int64_t n,
                std::vector<double>& out) {
  out.resize(static_cast<size_t>(H) * D);
  std::vector<double> row;
  for (int h = 0; h < H; ++h) {
    load_row(base, is_bf16, l * H + h, cap, D, n, row);
    for (int d = 0; d < D; ++d) out[static_cast<size_t>(h) * D + d] = row[d];
  }
}

// TaR and VaN of every past token of every layer with one index set per
// layer (Sec. 3.1, K in R^{H x N x D}): Eq. (tar) on the concatenated H*D key
// blocks, VaN the norm of the concatenated value block. k, v: [n_layers*H]
// [cap][D]; patch_id: [n_layers*H][cap] or NULL (the layer's first head's ids
// are used). tar_out, van_out: [n_layers][n_tokens], recent entries 0.
int oracle_scores_shared(const void* k, const void* v, int is_bf16, int64_t n_layers, int H,
                         int64_t cap, int D, int64_t n_tokens, int p, int r,
                         const uint16_t* patch_id, double* tar_out, double* van_out) {
  if (!k || !v || !tar_out || !van_out || n_layers < 0 || H <= 0 || D <= 0 || p <= 0 ||
      r <= 0 || n_tokens < 0 || n_tokens > cap || n_tokens % p != 0)
    return -1;
  const int64_t rp = static_cast<int64_t>(r) * p;
  if (rp > n_tokens) return -1;
  const int64_t n_past = n_tokens - rp;
  std::vector<double> kp, kr, vv;
  for (int64_t l = 0; l < n_layers; ++l) {
    double* tar = tar_out + l * n_tokens;
    double* van = van_out + l * n_tokens;
    for (int64_t n = 0; n < n_tokens; ++n) tar[n] = van[n] = 0.0;
    for (int64_t n = 0; n < n_past; ++n) {
      const int64_t q = patch_id ? patch_id[l * H * cap + n] : n % p;
      if (q < 0 || q >= p) return -1;
      load_token(k, is_bf16, l, H, cap, D, n, kp);
      double sum_cos = 0.0;
      for (int t = 0; t < r; ++t) {
        load_token(k, is_bf16, l, H, cap, D, n_past + static_cast<int64_t>(t) * p + q, kr);
        sum_cos += cosine(kp, kr);
      }
      tar[n] = -sum_cos / r;
      load_token(v, is_bf16, l, H, cap, D, n, vv);
      van[n] = l2norm(vv);
    }
  }
  return 0;
}

// VaN of every cached row of every layer, shared index set (the norm of the
// concatenated H x D value block). van_out: [n_layers][n_tokens].
int oracle_van_all_shared(const void* v, int is_bf16, int64_t n_layers, int H, int64_t cap, int D,
                          int64_t n_tokens, double* van_out) {
  if (!v || !van_out || n_layers < 0 || H <= 0 || D <= 0 || n_tokens < 0 || n_tokens > cap) return -1;
  std::vector<double> vv;
  for (int64_t l = 0; l < n_layers; ++l)
    for (int64_t n = 0; n < n_tokens; ++n) {
      load_token(v, is_bf16, l, H, cap, D, n, vv);
      van_out[l * n_tokens + n] = l2norm(vv);
    }
  return 0;
}

// Budget split used by the selection (Sec. 3.3, Algorithm 1 steps 3-5):
// out[0] = r p (recent tokens kept), out[1] = TaR picks among past tokens,
// out[2] = VaN picks among the remaining past tokens. The pass-through case
// (n_tokens <= budget) is reported as out = {-1,-1,-1}. Returns -1 when the
// arguments admit no selection (r p >= budget, alpha outside [0,1] or NaN).
int oracle_budget_split(int64_t n_tokens, int p, int r, int64_t budget,
                        double alpha, int64_t* out) {
  if (n_tokens <= budget) {
    out[0] = out[1] = out[2] = -1;
    return 0;
  }
  const int64_t rp = static_cast<int64_t>(r) * p;
  if (rp >= budget || alpha < 0.0 || alpha > 1.0 || !(alpha == alpha)) return -1;
  const int64_t tar_share = static_cast<int64_t>(std::floor(alpha * static_cast<double>(budget)));
  const int64_t n_tar = std::max<int64_t>(0, tar_share - rp);
  out[0] = rp;
  out[1] = n_tar;
  out[2] = budget - rp - n_tar;
  return 0;
}

// Selection (Algorithm 1 steps 3-5 with the Sec. 3.3 split). tar, van:
// [n_slabs][n_tokens] scores (recent entries ignored). kept_out:
// [n_slabs][budget], ascending per slab; in the pass-through case
// (n_tokens <= budget) it is 0..n_tokens-1 followed by -1.
// gaps_out (optional, [n_slabs][2]): per stage the score gap between the last
// token taken and the first token left, |s_(k) - s_(k+1)|; the VaN entry is
// relative to |s_(k)|. +inf when the stage has nothing to decide.
int oracle_select(const double* tar, const double* van, int64_t n_slabs,
                  int64_t n_tokens, int p, int r, int64_t budget, double alpha,
                  int32_t* kept_out, double* gaps_out) {
  int64_t split[3];
  if (!tar || !van || !kept_out || p <= 0 || r <= 0 || budget <= 0) return -1;
  if (oracle_budget_split(n_tokens, p, r, budget, alpha, split) != 0) return -1;
  const double inf = std::numeric_limits<double>::infinity();
  for (int64_t s = 0; s < n_slabs; ++s) {
    int32_t* kept = kept_out + s * budget;
    if (split[0] < 0) {  // pass-through: nothing to evict
      for (int64_t j = 0; j < budget; ++j) kept[j] = j < n_tokens ? static_cast<int32_t>(j) : -1;
      if (gaps_out) gaps_out[2 * s] = gaps_out[2 * s + 1] = inf;
      continue;
    }
    const double* ts = tar + s * n_tokens;
    const double* vs = van + s * n_tokens;
    const int64_t rp = split[0], n_tar = split[1], n_van = split[2];
    const int64_t n_past = n_tokens - rp;

    // TaR stage: order past tokens by (s_TaR desc, index asc).
    std::vector<int64_t> past(n_past);
    for (int64_t n = 0; n < n_past; ++n) past[n] = n;
    std::vector<int64_t> by_tar = past;
    std::sort(by_tar.begin(), by_tar.end(), [&](int64_t a, int64_t b) {
      return ranks_above(ts[a], a, ts[b], b);
    });
    std::vector<char> keep(n_tokens, 0);
    for (int64_t n = n_past; n < n_tokens; ++n) keep[n] = 1;  // recent frames
    for (int64_t i = 0; i < n_tar; ++i) keep[by_tar[i]] = 1;
    double gap_tar = inf;
    if (n_tar > 0 && n_tar < n_past)
      gap_tar = std::fabs(ts[by_tar[n_tar - 1]] - ts[by_tar[n_tar]]);

    // VaN stage: among past tokens TaR did not take, (s_VaN desc, index asc).
    std::vector<int64_t> rest;
    for (int64_t n = 0; n < n_past; ++n)
      if (!keep[n]) rest.push_back(n);
    std::sort(rest.begin(), rest.end(), [&](int64_t a, int64_t b) {
      return ranks_above(vs[a], a, vs[b], b);
    });
    for (int64_t i = 0; i < n_van; ++i) keep[rest[i]] = 1;
    double gap_van = inf;
    const int64_t n_rest = static_cast<int64_t>(rest.size());
    if (n_van > 0 && n_van < n_rest) {
      const double a = vs[rest[n_van - 1]], b = vs[rest[n_van]];
      gap_van = std::fabs(a - b) / std::max(std::fabs(a), 1e-300);
    }

    int64_t j = 0;
    for (int64_t n = 0; n < n_tokens; ++n)
      if (keep[n]) kept[j++] = static_cast<int32_t>(n);
    if (j != budget) return -2;  // cannot happen: the split sums to budget
    if (gaps_out) {
      gaps_out[2 * s] = gap_tar;
      gaps_out[2 * s + 1] = gap_van;
    }
  }
  return 0;
}

// Compaction (Sec. 3.1; Algorithm 2 last step): dst[s][j] = src[s][kept[s][j]]
// row by row, bytes copied unchanged. Rows with kept == -1 are left untouched.
int oracle_gather_rows(const void* src, void* dst, int64_t row_bytes,
                       int64_t n_slabs, int64_t cap_src, int64_t cap_dst,
                       const int32_t* kept, int64_t budget) {
  if (!src || !dst || !kept || row_bytes <= 0) return -1;
  const char* s8 = static_cast<const char*>(src);
  char* d8 = static_cast<char*>(dst);
  for (int64_t s = 0; s < n_slabs; ++s)
    for (int64_t j = 0; j < budget; ++j) {
      const int32_t n = kept[s * budget + j];
      if (n < 0) continue;
      if (n >= cap_src || j >= cap_dst) return -1;
      std::memcpy(d8 + (s * cap_dst + j) * row_bytes, s8 + (s * cap_src + n) * row_bytes,
                  static_cast<size_t>(row_bytes));
    }
  return 0;
}

// Patch ids travel with their tokens: dst[s][j] = src ? src[s][kept] : kept mod p.
int oracle_gather_patch(const uint16_t* src_pid, uint16_t* dst_pid, int64_t n_slabs,
                        int64_t cap_src, int64_t cap_dst, int p,
                        const int32_t* kept, int64_t budget) {
  if (!dst_pid || !kept || p <= 0) return -1;
  for (int64_t s = 0; s < n_slabs; ++s)
    for (int64_t j = 0; j < budget; ++j) {
      const int32_t n = kept[s * budget + j];
      if (n < 0) continue;
      dst_pid[s * cap_dst + j] =
          src_pid ? src_pid[s * cap_src + n] : static_cast<uint16_t>(n % p);
    }
  return 0;
}

// Frame ids travel with their tokens: dst[s][j] = src ? src[s][kept] : kept div p.
int oracle_gather_frame(const uint32_t* src_fid, uint32_t* dst_fid, int64_t n_slabs,
                        int64_t cap_src, int64_t cap_dst, int p,
                        const int32_t* kept, int64_t budget) {
  if (!dst_fid || !kept || p <= 0) return -1;
  for (int64_t s = 0; s < n_slabs; ++s)
    for (int64_t j = 0; j < budget; ++j) {
      const int32_t n = kept[s * budget + j];
      if (n < 0) continue;
      dst_fid[s * cap_dst + j] =
          src_fid ? src_fid[s * cap_src + n] : static_cast<uint32_t>(n / p);
    }
  return 0;
}

// VaN of every cached row, recent frames included (Algorithm 2 takes mu and
// sigma over the whole layer's ||V_l||_2). van_out: [n_slabs][n_tokens].
int oracle_van_all(const void* v, int is_bf16, int64_t n_slabs, int64_t cap, int D,
                   int64_t n_tokens, double* van_out) {
  if (!v || !van_out || n_slabs < 0 || D <= 0 || n_tokens < 0 || n_tokens > cap) return -1;
  std::vector<double> vv;
  for (int64_t s = 0; s < n_slabs; ++s)
    for (int64_t n = 0; n < n_tokens; ++n) {
      load_row(v, is_bf16, s, cap, D, n, vv);
      van_out[s * n_tokens + n] = l2norm(vv);
    }
  return 0;
}

// Pool size g(CV) of Algorithm 2: 7 if CV < tau_1, 5 if tau_1 <= CV < tau_2,
// 3 if tau_2 <= CV < tau_3, 1 if CV >= tau_3. A NaN CV satisfies none of the
// strict comparisons and gets 1 (no pooling).
int oracle_pool_size(double cv, const double* tau) {
  if (cv < tau[0]) return 7;
  if (cv < tau[1]) return 5;
  if (cv < tau[2]) return 3;
  return 1;
}

// Layer-adaptive pooling of VaN (Sec. 3.2; Algorithm 2). van: [n_slabs][n_tokens]
// VaN of every cached row; slabs s = l * n_kv_heads + h form layer l.
// patch_id (uint16) and frame_id (uint32), both [n_slabs][id_stride] or both
// NULL (then row n is patch n mod p of frame n div p). For each layer:
//   mu = mean, sigma = population std of all its heads' VaN values,
//   CV = sigma / mu, k = g(CV);
// for each row n of each of its slabs, at frame F and grid position (i, j)
// (patch q = i * grid_w + j):
//   k == 1: pooled = VaN[n];
//   k  > 1: pooled = mean of VaN[m] over the rows m of the same slab and
//           frame F whose position (i', j') has |i' - i| <= k div 2 and
//           |j' - j| <= k div 2 (row n itself included);
//   a patch id >= p has no position: its pooled value is NaN (k > 1).
// pooled_out: [n_slabs][n_tokens]; pool_size_out, cv_out: [n_layers] or NULL.
int oracle_van_pool(const double* van, int64_t n_slabs, int n_kv_heads, int64_t n_tokens,
                    int grid_h, int grid_w, const uint16_t* patch_id,
                    const uint32_t* frame_id, int64_t id_stride, const double* tau,
                    double* pooled_out, int32_t* pool_size_out, double* cv_out) {
  if (!van || !pooled_out || !tau || n_kv_heads <= 0 || n_slabs % n_kv_heads != 0 ||
      n_tokens <= 0 || grid_h <= 0 || grid_w <= 0 || (patch_id == nullptr) != (frame_id == nullptr) ||
      (patch_id && id_stride < n_tokens))
    return -1;
  const int64_t p = static_cast<int64_t>(grid_h) * grid_w;
  const double nan = std::numeric_limits<double>::quiet_NaN();
  const int64_t n_layers = n_slabs / n_kv_heads;
  for (int64_t l = 0; l < n_layers; ++l) {
    const double* lv = van + l * n_kv_heads * n_tokens;
    const int64_t count = n_kv_heads * n_tokens;
    double sum = 0.0;
    for (int64_t i = 0; i < count; ++i) sum += lv[i];
    const double mu = sum / static_cast<double>(count);
    double ss = 0.0;
    for (int64_t i = 0; i < count; ++i) ss += (lv[i] - mu) * (lv[i] - mu);
    const double sigma = std::sqrt(ss / static_cast<double>(count));
    const double cv = sigma / mu;
    const int k = oracle_pool_size(cv, tau);
    if (pool_size_out) pool_size_out[l] = k;
    if (cv_out) cv_out[l] = cv;
    const int64_t half = k / 2;
    for (int64_t h = 0; h < n_kv_heads; ++h) {
      const int64_t s = l * n_kv_heads + h;
      const double* sv = van + s * n_tokens;
      double* out = pooled_out + s * n_tokens;
      if (k == 1) {
        for (int64_t n = 0; n < n_tokens; ++n) out[n] = sv[n];
        continue;
      }
      std::vector<int64_t> frame(n_tokens), patch(n_tokens);
      std::map<int64_t, std::vector<int64_t>> rows_of_frame;
      for (int64_t n = 0; n < n_tokens; ++n) {
        frame[n] = patch_id ? static_cast<int64_t>(frame_id[s * id_stride + n]) : n / p;
        patch[n] = patch_id ? static_cast<int64_t>(patch_id[s * id_stride + n]) : n % p;
        rows_of_frame[frame[n]].push_back(n);
      }
      for (int64_t n = 0; n < n_tokens; ++n) {
        if (patch[n] >= p) {
          out[n] = nan;
          continue;
        }
        const int64_t i = patch[n] / grid_w, j = patch[n] % grid_w;
        double acc = 0.0;
        int64_t cnt = 0;
        for (int64_t m : rows_of_frame[frame[n]]) {
          if (patch[m] >= p) continue;
          const int64_t im = patch[m] / grid_w, jm = patch[m] % grid_w;
          if (std::llabs(im - i) <= half && std::llabs(jm - j) <= half) {
            acc += sv[m];
            ++cnt;
          }
        }
        out[n] = acc / static_cast<double>(cnt);
      }
    }
  }
  return 0;
}

// Frame-level TaR ("TaR Frame" ablation): every past row n of every unit
// gets the mean of tar over the past rows of its frame (frame_id with
// stride id_stride if given, else n div p). tar: [units][n_tokens], in place.
int oracle_frame_mean(double* tar, int64_t units, int64_t n_tokens, int64_t n_past, int p,
                      const uint32_t* frame_id, int64_t id_stride) {
  if (!tar || p <= 0 || n_past < 0 || n_past > n_tokens) return -1;
  for (int64_t u = 0; u < units; ++u) {
    double* t = tar + u * n_tokens;
    std::map<int64_t, std::pair<double, int64_t>> acc;  // frame -> (sum, count)
    std::vector<int64_t> frame(n_past);
    for (int64_t n = 0; n < n_past; ++n) {
      frame[n] = frame_id ? static_cast<int64_t>(frame_id[u * id_stride + n]) : n / p;
      acc[frame[n]].first += t[n];
      acc[frame[n]].second += 1;
    }
    for (int64_t n = 0; n < n_past; ++n) {
      const auto& a = acc[frame[n]];
      t[n] = a.first / static_cast<double>(a.second);
    }
  }
  return 0;
}

// Uniform Select: for each of n_units units, the rows of the k = budget / p
// whole frames F - 1 - floor(i F / k), i = 0..k-1, of the F = n_tokens / p
// frames (p consecutive rows each), ascending. budget must be a multiple of p
// below n_tokens.
int oracle_uniform_select(int64_t n_units, int64_t n_tokens, int p, int64_t budget,
                          int32_t* kept_out) {
  if (!kept_out || p <= 0 || n_tokens % p != 0 || budget % p != 0 || budget <= 0 ||
      budget >= n_tokens)
    return -1;
  const int64_t F = n_tokens / p, k = budget / p;
  std::vector<int64_t> frames;
  for (int64_t i = 0; i < k; ++i) frames.push_back(F - 1 - (i * F) / k);
  std::sort(frames.begin(), frames.end());
  for (int64_t u = 0; u < n_units; ++u) {
    int32_t* kept = kept_out + u * budget;
    int64_t j = 0;
    for (int64_t f : frames)
      for (int q = 0; q < p; ++q) kept[j++] = static_cast<int32_t>(f * p + q);
  }
  return 0;
}

// One whole pass over slabs [0, n_slabs): scores, selection, compaction of K
// and V (and of patch ids when dst_pid != NULL, of frame ids when dst_fid !=
// NULL). With van_pool != 0 the VaN stage ranks the layer-adaptive pooled
// VaN (tau: the three CV thresholds; n_kv_heads groups slabs into layers;
// src_fid goes with src_pid). pool_size_out: [n_slabs / n_kv_heads] or NULL.
// With shared != 0 one index set per layer is chosen (scores of the
// concatenated head blocks) and kept_out is [n_slabs / n_kv_heads][budget].
// ablation: 0 none, 1 TaR Reverse, 2 VaN Reverse, 3 TaR Frame, 4 Uniform
// Select (no scores; budget a multiple of p).
int oracle_compress(const void* k, const void* v, int is_bf16, int64_t n_slabs,
                    int64_t cap, int D, int64_t n_tokens, int p, int r,
                    int64_t budget, double alpha, const uint16_t* src_pid,
                    void* k_dst, void* v_dst, uint16_t* dst_pid, int32_t* kept_out,
                    int van_pool, const double* tau, int n_kv_heads, int grid_w,
                    const uint32_t* src_fid, uint32_t* dst_fid, int32_t* pool_size_out,
                    int shared, int ablation) {
  // With a shared index set the scores, the selection and kept_out are per
  // layer ("units" = layers); else per slab.
  if (n_kv_heads <= 0 || n_slabs % n_kv_heads != 0) return -1;
  const int64_t H = shared ? n_kv_heads : 1;
  const int64_t units = n_slabs / H;
  std::vector<double> tar(static_cast<size_t>(units * n_tokens));
  std::vector<double> van(tar.size());
  if (n_tokens > budget && ablation != 4) {
    const int rc = shared ? oracle_scores_shared(k, v, is_bf16, units, static_cast<int>(H), cap, D,
                                                 n_tokens, p, r, src_pid, tar.data(), van.data())
                          : oracle_scores(k, v, is_bf16, n_slabs, cap, D, n_tokens, p, r, src_pid,
                                          tar.data(), van.data());
    if (rc != 0) return -1;
    const int64_t n_past = n_tokens - static_cast<int64_t>(r) * p;
    if (ablation == 3 && src_pid && !src_fid) return -1;  // frames need frame ids once compacted
    if (ablation == 3 &&  // TaR Frame: a unit's ids are those of its first head
        oracle_frame_mean(tar.data(), units, n_tokens, n_past, p, src_pid ? src_fid : nullptr,
                          cap * H) != 0)
      return -1;
    if (van_pool) {
      if (grid_w <= 0 || p % grid_w != 0) return -1;
      std::vector<double> all(tar.size());
      const int rv = shared ? oracle_van_all_shared(v, is_bf16, units, static_cast<int>(H), cap, D,
                                                    n_tokens, all.data())
                            : oracle_van_all(v, is_bf16, n_slabs, cap, D, n_tokens, all.data());
      if (rv != 0) return -1;
      // A layer is one unit of H heads, or (shared) one unit on its own; the
      // ids of a shared unit are those of its first head.
      if (oracle_van_pool(all.data(), units, shared ? 1 : n_kv_heads, n_tokens, p / grid_w,
                          grid_w, src_pid, src_fid, cap * H, tau, van.data(), pool_size_out,
                          nullptr) != 0)
        return -1;
    }
  }
  int32_t* kept_sel = kept_out;
  if (ablation == 1)  // TaR Reverse: the lowest TaR first
    for (double& x : tar) x = -x;
  if (ablation == 2)  // VaN Reverse: the lowest VaN first
    for (double& x : van) x = -x;
  if (ablation == 4 && n_tokens > budget) {
    if (oracle_uniform_select(units, n_tokens, p, budget, kept_sel) != 0) return -1;
  } else if (oracle_select(tar.data(), van.data(), units, n_tokens, p, r, budget, alpha,
                           kept_sel, nullptr) != 0) {
    return -1;
  }
  if (n_tokens <= budget) return 0;  // pass-through leaves the cache as it is
  // Every head of a unit is compacted with the unit's indices.
  std::vector<int32_t> kept_slab(static_cast<size_t>(n_slabs * budget));
  for (int64_t s = 0; s < n_slabs; ++s)
    for (int64_t j = 0; j < budget; ++j) kept_slab[s * budget + j] = kept_sel[(s / H) * budget + j];
  const int32_t* kept = kept_slab.data();
  const int64_t row_bytes = static_cast<int64_t>(D) * (is_bf16 ? 2 : 4);
  if (oracle_gather_rows(k, k_dst, row_bytes, n_slabs, cap, cap, kept, budget) != 0) return -1;
  if (oracle_gather_rows(v, v_dst, row_bytes, n_slabs, cap, cap, kept, budget) != 0) return -1;
  if (dst_pid && oracle_gather_patch(src_pid, dst_pid, n_slabs, cap, cap, p, kept, budget) != 0)
    return -1;
  if (dst_fid && oracle_gather_frame(src_fid, dst_fid, n_slabs, cap, cap, p, kept, budget) != 0)
    return -1;
  return 0;
}

}  // extern "C"
