// C ABI of libipv.so (declared in include/ipv.h): state, argument checks,
// kernel sequencing and optional per-kernel event timing.
#include <cmath>
#include <cstddef>
#include <cstdarg>
#include <cstdio>
#include <ctime>
#include <string>
#include <vector>

#include "ipv.h"
#include "ipv_common.cuh"

static_assert(ipv::kMaxTokens == IPV_MAX_TOKENS, "selection shared-memory limit");
static_assert(ipv::kMaxPoolFrame == IPV_MAX_POOL_FRAME_TOKENS, "pooling shared-memory limit");

namespace {

struct EventPair {
  cudaEvent_t start = nullptr, stop = nullptr;
};

struct State {
  bool ready = false;
  ipv_options opt{};
  int num_sms = 0;
  float* tar = nullptr;   // [max_slabs][token_capacity]
  float* van = nullptr;
  float* m = nullptr;     // [max_slabs][max_frame_tokens][max_head_dim]
  float* pooled = nullptr;  // [max_slabs][token_capacity], van_pool only
  float* kk = nullptr;      // [max_slabs][token_capacity], head_shared only: per-head |k|^2
  float* tar_l = nullptr;   // [max_slabs][token_capacity], head_shared only: per-layer scores
  float* van_l = nullptr;
  ipv::WinState* wstate = nullptr;
  unsigned* wflags = nullptr;  // [kWinFlags][max_slabs]
  unsigned* claim = nullptr;   // [3] compaction work counters, zero between passes
  bool win_dirty = false;      // a failed launch may have left counters behind
  int64_t wait_limit = int64_t{1} << 20;  // polls before a wait of the fused pass gives up
  bool profiling = false;
  std::vector<EventPair> pool;                      // idle event pairs
  std::vector<EventPair> pending[IPV_NUM_KERNELS];  // recorded, not yet read
};

State g;
thread_local std::string g_err;

void free_scratch(State& s) {
  for (void* p : {static_cast<void*>(s.tar), static_cast<void*>(s.van), static_cast<void*>(s.m),
                  static_cast<void*>(s.pooled), static_cast<void*>(s.kk), static_cast<void*>(s.tar_l),
                  static_cast<void*>(s.van_l), static_cast<void*>(s.wstate), static_cast<void*>(s.wflags),
                  static_cast<void*>(s.claim)})
    cudaFree(p);
}

ipv_status fail(ipv_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  g_err = std::string(ipv_status_string(s)) + ": " + buf;
  return s;
}

ipv_status cuda_fail(cudaError_t e, const char* what) {
  return fail(IPV_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int elem_bytes() { return g.opt.dtype == IPV_BF16 ? 2 : 4; }

int default_recent_frames(int64_t f) {
  if (g.opt.recent_frames > 0) return g.opt.recent_frames;
  const int64_t r = static_cast<int64_t>(std::floor(static_cast<double>(f) / 8.0 + 0.5));
  return static_cast<int>(r < 1 ? 1 : r);
}

// ------------------------------------------------------------------ profiling
EventPair take_pair() {
  if (!g.pool.empty()) {
    EventPair p = g.pool.back();
    g.pool.pop_back();
    return p;
  }
  EventPair p;
  cudaEventCreate(&p.start);
  cudaEventCreate(&p.stop);
  return p;
}

void prof_begin(int id, cudaStream_t st) {
  if (!g.profiling) return;
  EventPair p = take_pair();
  cudaEventRecord(p.start, st);
  g.pending[id].push_back(p);
}

void prof_end(int id, cudaStream_t st) {
  if (!g.profiling || g.pending[id].empty()) return;
  cudaEventRecord(g.pending[id].back().stop, st);
}

void release_events() {
  for (auto& v : g.pending) {
    for (auto& p : v) g.pool.push_back(p);
    v.clear();
  }
  for (auto& p : g.pool) {
    cudaEventDestroy(p.start);
    cudaEventDestroy(p.stop);
  }
  g.pool.clear();
}

// ------------------------------------------------------------- argument checks
struct Shape {
  int64_t S, N, f;
  int D, p, r;
  int64_t rp;
};

// Checks that need no library state; then the init check; then the rest.
ipv_status check_cache(const ipv_kv* k, const ipv_kv* v, int L, int H, int D, int64_t N, int gh,
                       int gw, bool need_dst, Shape* sh) {
  if (!k || !v) return fail(IPV_EINVAL, "k and v must not be NULL");
  if (k->cur != 0 && k->cur != 1) return fail(IPV_EINVAL, "k->cur must be 0 or 1");
  if (v->cur != 0 && v->cur != 1) return fail(IPV_EINVAL, "v->cur must be 0 or 1");
  if (L <= 0 || H <= 0 || D <= 0 || N <= 0 || gh <= 0 || gw <= 0)
    return fail(IPV_EINVAL, "sizes must be positive (layers %d heads %d head_dim %d tokens %lld grid %dx%d)",
                L, H, D, static_cast<long long>(N), gh, gw);
  const int64_t p = static_cast<int64_t>(gh) * gw;
  if (p > 65535) return fail(IPV_EINVAL, "frame_grid_h*frame_grid_w = %lld exceeds 65535", static_cast<long long>(p));
  if (N % p != 0)
    return fail(IPV_EINVAL, "n_tokens %lld is not a multiple of the %lld tokens of a frame",
                static_cast<long long>(N), static_cast<long long>(p));
  const void* src_k = k->buf[k->cur];
  const void* src_v = v->buf[v->cur];
  if (!src_k || !src_v) return fail(IPV_EINVAL, "live cache halves buf[cur] must not be NULL");
  if (!aligned16(src_k) || !aligned16(src_v)) return fail(IPV_EINVAL, "cache halves must be 16-byte aligned");
  if (src_k == src_v) return fail(IPV_EINVAL, "k and v share one buffer");
  if (need_dst) {
    const void* dk = k->buf[1 - k->cur];
    const void* dv = v->buf[1 - v->cur];
    if (!dk || !dv) return fail(IPV_EINVAL, "destination halves buf[1-cur] must not be NULL");
    if (!aligned16(dk) || !aligned16(dv)) return fail(IPV_EINVAL, "cache halves must be 16-byte aligned");
    if (dk == src_k || dv == src_v || dk == src_v || dv == src_k || dk == dv)
      return fail(IPV_EINVAL, "ping-pong halves must be distinct buffers");
    const uint16_t* ps = k->patch_id[k->cur];
    const uint16_t* pd = k->patch_id[1 - k->cur];
    if (pd && pd == ps) return fail(IPV_EINVAL, "patch-id halves must be distinct buffers");
    const uint32_t* fs = k->frame_id[k->cur];
    const uint32_t* fd = k->frame_id[1 - k->cur];
    if (fd && fd == fs) return fail(IPV_EINVAL, "frame-id halves must be distinct buffers");
    if (fd && (reinterpret_cast<uintptr_t>(fd) & 3u)) return fail(IPV_EINVAL, "frame ids must be 4-byte aligned");
  }
  const uint32_t* fsrc = k->frame_id[k->cur];
  if (fsrc && (reinterpret_cast<uintptr_t>(fsrc) & 3u)) return fail(IPV_EINVAL, "frame ids must be 4-byte aligned");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  const int64_t S = static_cast<int64_t>(L) * H;
  if (S > g.opt.max_slabs)
    return fail(IPV_EINVAL, "n_layers*n_kv_heads = %lld exceeds max_slabs %lld", static_cast<long long>(S),
                static_cast<long long>(g.opt.max_slabs));
  if (D > g.opt.max_head_dim) return fail(IPV_EINVAL, "head_dim %d exceeds max_head_dim %d", D, g.opt.max_head_dim);
  if ((static_cast<int64_t>(D) * elem_bytes()) % 16 != 0)
    return fail(IPV_EINVAL, "head_dim*element size must be a multiple of 16 bytes");
  if (p > g.opt.max_frame_tokens)
    return fail(IPV_EINVAL, "frame tokens %lld exceed max_frame_tokens %d", static_cast<long long>(p),
                g.opt.max_frame_tokens);
  if (N > g.opt.token_capacity)
    return fail(IPV_EINVAL, "n_tokens %lld exceeds token_capacity %lld", static_cast<long long>(N),
                static_cast<long long>(g.opt.token_capacity));
  sh->S = S;
  sh->N = N;
  sh->D = D;
  sh->p = static_cast<int>(p);
  sh->f = N / p;
  sh->r = default_recent_frames(sh->f);
  sh->rp = static_cast<int64_t>(sh->r) * p;
  return IPV_OK;
}

// Budget split of Sec. 3.3 / Algorithm 1: floor(alpha C) for TaR including the
// r p recent tokens, the rest of C for VaN.
void split_budget(int64_t budget, float tar_ratio, int64_t rp, int64_t* n_tar, int64_t* n_van) {
  const int64_t share = static_cast<int64_t>(std::floor(static_cast<double>(tar_ratio) * budget));
  *n_tar = share > rp ? share - rp : 0;
  *n_van = budget - rp - *n_tar;
}

ipv_status check_select_args(int64_t N, int64_t budget, float tar_ratio, const int32_t* kept) {
  if (!kept) return fail(IPV_EINVAL, "kept_idx_out must not be NULL");
  if ((reinterpret_cast<uintptr_t>(kept) & 3u) != 0) return fail(IPV_EINVAL, "kept_idx_out must be 4-byte aligned");
  if (budget <= 0) return fail(IPV_EINVAL, "budget must be positive");
  if (!(tar_ratio >= 0.0f && tar_ratio <= 1.0f)) return fail(IPV_EINVAL, "tar_ratio must lie in [0, 1]");
  if (budget > INT32_MAX || N > INT32_MAX) return fail(IPV_EINVAL, "sizes exceed int32 indices");
  return IPV_OK;
}

ipv_status after_launch(cudaError_t e, const char* what) {
  return e == cudaSuccess ? IPV_OK : cuda_fail(e, what);
}

// The "TaR Frame" ablation: each past row of each unit (slab, or layer with
// the shared index set, whose ids are its first head's) takes its frame's
// mean TaR.
cudaError_t launch_tar_frame(float* tar, const ipv_kv* k, int64_t units, int hsh, const Shape& sh,
                             cudaStream_t st) {
  ipv::FrameMeanArgs fa{};
  fa.tar = tar;
  fa.frame_id = k->patch_id[k->cur] ? k->frame_id[k->cur] : nullptr;
  fa.id_stride = g.opt.token_capacity * hsh;
  fa.units = units;
  fa.n_tokens = sh.N;
  fa.n_past = sh.N - sh.rp;
  fa.p = sh.p;
  return ipv::launch_frame_mean(fa, st);
}

// The shared index set reads a token's n_kv_heads head-rows as one block
// (at most 128 16-byte chunks per lane group of the recent-frame mean).
ipv_status check_shared(int n_kv_heads, int head_dim) {
  if (static_cast<int64_t>(n_kv_heads) * head_dim * elem_bytes() > 2048)
    return fail(IPV_EINVAL, "head_shared needs n_kv_heads*head_dim*element size <= 2048 bytes");
  return IPV_OK;
}

// Steps (i)-(ii) with one index set per layer: the recent-frame mean of each
// layer's head blocks, the heads' partial sums, and their combination into
// per-layer TaR and VaN ([L][n_tokens] in tar_out, van_out).
cudaError_t launch_shared_scores(const ipv::ScoreArgs& phys, int n_kv_heads, float* tar_out,
                                 float* van_out, int zero_recent, cudaStream_t st) {
  ipv::ScoreArgs am = phys;  // the layer view of the recent-frame mean
  am.n_slabs = phys.n_slabs / n_kv_heads;
  am.hs = n_kv_heads;
  am.tar = tar_out;
  am.van = van_out;
  am.zero_recent = zero_recent;
  am.van_recent = g.opt.van_pool;
  am.kk = nullptr;
  ipv::ScoreArgs a = phys;   // per head-slab partial sums into scratch
  a.tar = g.tar;
  a.van = g.van;
  a.kk = g.kk;
  a.zero_recent = 0;
  a.van_recent = 0;
  a.hs = 1;
  prof_begin(0, st);
  cudaError_t e = ipv::launch_recent_mean(am, st);
  prof_end(0, st);
  if (e != cudaSuccess) return e;
  prof_begin(1, st);
  e = ipv::launch_score(a, st);
  prof_end(1, st);
  if (e != cudaSuccess) return e;
  ipv::CombineArgs c{};
  c.dot = g.tar;
  c.kk = g.kk;
  c.vv = g.van;
  c.tar = tar_out;
  c.van = van_out;
  c.n_layers = am.n_slabs;
  c.n_tokens = phys.n_tokens;
  c.n_past = phys.n_tokens - static_cast<int64_t>(phys.r) * phys.p;
  c.hs = n_kv_heads;
  c.num_sms = g.num_sms;
  prof_begin(6, st);
  e = ipv::launch_combine(c, st);
  prof_end(6, st);
  return e;
}

// Work decomposition of the fused pass (window.cu). Tuning constants: score
// items of at most IPV_WIN_PATCHES patches, gather items of IPV_WIN_ROWS
// selected rows, and a window of IPV_WIN_LAG slabs that scoring may run ahead
// of compaction (the L2 holds about that many slabs' rows).
#ifndef IPV_WIN_PATCHES
#define IPV_WIN_PATCHES 16
#endif
#ifndef IPV_WIN_ROWS
#define IPV_WIN_ROWS 512
#endif
#ifndef IPV_WIN_LAG
#define IPV_WIN_LAG 8
#endif

size_t fused_smem(const ipv::WinArgs& w) {
  return ipv::window_smem_bytes(w.qmax, w.sc.D, w.sc.is_bf16 ? 2 : 4, w.sc.r,
                                w.sc.n_tokens - static_cast<int64_t>(w.sc.r) * w.sc.p);
}

// Fills the fused pass's arguments; false if the pass does not fit it (the
// selection's keys in the registers of one block, a score item's recent rows
// in shared memory that leaves room for a second block on the SM).
bool fused_args(const ipv::ScoreArgs& a, const ipv::SelectArgs& sa, const ipv::GatherArgs& ga,
                const Shape& sh, int64_t budget, ipv::WinArgs* w) {
  const int64_t n_past = sh.N - sh.rp;
  if (n_past > static_cast<int64_t>(ipv::kWinBlock) * ipv::kWinRegE) return false;
  w->sc = a;
  w->se = sa;
  w->ga = ga;
  w->state = g.wstate;
  w->flags = g.wflags;
  w->n_si = (sh.p + IPV_WIN_PATCHES - 1) / IPV_WIN_PATCHES;
  w->qmax = (sh.p + w->n_si - 1) / w->n_si;
  while (w->qmax > 1 && fused_smem(*w) > ipv::kWinSmemMax) {  // fewer patches per item for wide rows
    w->n_si = (sh.p + w->qmax - 2) / (w->qmax - 1);
    w->qmax = (sh.p + w->n_si - 1) / w->n_si;
  }
  w->rows_gi = IPV_WIN_ROWS;
  w->n_gi = static_cast<int>((budget - sh.rp + IPV_WIN_ROWS - 1) / IPV_WIN_ROWS);
  w->lag = IPV_WIN_LAG;
  w->n_stream = g.num_sms;
  w->n_owner = static_cast<int>(sh.S < g.num_sms ? sh.S : g.num_sms);
  w->spin_limit = g.wait_limit;
  if (fused_smem(*w) > ipv::kWinSmemMax) return false;
  int per_sm = 0;
  if (ipv::window_blocks_per_sm(*w, fused_smem(*w), &per_sm) != cudaSuccess || per_sm < 2) {
    cudaGetLastError();
    return false;
  }
  return true;
}

}  // namespace

namespace ipv {
// Lets other translation units of the library report through ipv_last_error.
void record_error(ipv_status s, const char* msg) { fail(s, "%s", msg); }
}  // namespace ipv

extern "C" {

const char* ipv_status_string(ipv_status s) {
  switch (s) {
    case IPV_OK: return "IPV_OK";
    case IPV_EINVAL: return "IPV_EINVAL";
    case IPV_ENOINIT: return "IPV_ENOINIT";
    case IPV_ENOMEM: return "IPV_ENOMEM";
    case IPV_ECUDA: return "IPV_ECUDA";
    case IPV_ETIMEOUT: return "IPV_ETIMEOUT";
  }
  return "IPV_UNKNOWN";
}

const char* ipv_last_error(void) { return g_err.c_str(); }

void ipv_shutdown(void) {
  if (!g.ready) return;
  cudaSetDevice(g.opt.device);
  cudaDeviceSynchronize();
  release_events();
  free_scratch(g);
  g = State{};
}

ipv_status ipv_init(const ipv_options* opt) {
  if (!opt) return fail(IPV_EINVAL, "options must not be NULL");
  if (opt->dtype != IPV_BF16 && opt->dtype != IPV_F32) return fail(IPV_EINVAL, "unknown dtype %d", opt->dtype);
  if (opt->device < 0) return fail(IPV_EINVAL, "device must be >= 0");
  if (opt->recent_frames < 0) return fail(IPV_EINVAL, "recent_frames must be >= 0");
  if (opt->max_head_dim <= 0 || opt->max_head_dim > 512) return fail(IPV_EINVAL, "max_head_dim must be in [1, 512]");
  if (opt->max_frame_tokens <= 0 || opt->max_frame_tokens > 65535)
    return fail(IPV_EINVAL, "max_frame_tokens must be in [1, 65535]");
  if (opt->max_slabs <= 0 || opt->max_slabs > INT32_MAX) return fail(IPV_EINVAL, "max_slabs must be in [1, 2^31)");
  if (opt->token_capacity <= 0 || opt->token_capacity > INT32_MAX)
    return fail(IPV_EINVAL, "token_capacity must be in [1, 2^31)");
  if (opt->single_kernel != 0 && opt->single_kernel != 1)
    return fail(IPV_EINVAL, "single_kernel must be 0 or 1");
  if (opt->van_pool != 0 && opt->van_pool != 1) return fail(IPV_EINVAL, "van_pool must be 0 or 1");
  if (opt->head_shared != 0 && opt->head_shared != 1) return fail(IPV_EINVAL, "head_shared must be 0 or 1");
  if (opt->head_shared && opt->single_kernel)
    return fail(IPV_EINVAL, "head_shared runs with the step kernels only (single_kernel = 0)");
  if (opt->ablation < IPV_ABLATION_NONE || opt->ablation > IPV_ABLATION_UNIFORM)
    return fail(IPV_EINVAL, "unknown ablation %d", opt->ablation);
  if (opt->ablation != IPV_ABLATION_NONE && opt->single_kernel)
    return fail(IPV_EINVAL, "ablation variants run with the step kernels only (single_kernel = 0)");
  if (opt->ablation == IPV_ABLATION_TAR_FRAME && opt->max_frame_tokens > IPV_MAX_POOL_FRAME_TOKENS)
    return fail(IPV_EINVAL, "the frame-level TaR needs max_frame_tokens <= %d", IPV_MAX_POOL_FRAME_TOKENS);
  if (opt->van_pool) {
    if (opt->single_kernel) return fail(IPV_EINVAL, "van_pool runs with the step kernels only (single_kernel = 0)");
    if (opt->max_frame_tokens > IPV_MAX_POOL_FRAME_TOKENS)
      return fail(IPV_EINVAL, "van_pool needs max_frame_tokens <= %d", IPV_MAX_POOL_FRAME_TOKENS);
    const float* t = opt->cv_tau;
    if (t[0] != t[0] || t[1] != t[1] || t[2] != t[2] || !(t[0] <= t[1] && t[1] <= t[2]))
      return fail(IPV_EINVAL, "cv_tau must be ordered tau_1 <= tau_2 <= tau_3 (no NaN)");
  }
  ipv_shutdown();
  int n_dev = 0;
  cudaError_t e = cudaGetDeviceCount(&n_dev);
  if (e != cudaSuccess) return cuda_fail(e, "cudaGetDeviceCount");
  if (opt->device >= n_dev) return fail(IPV_EINVAL, "device %d not present (%d devices)", opt->device, n_dev);
  if ((e = cudaSetDevice(opt->device)) != cudaSuccess) return cuda_fail(e, "cudaSetDevice");
  cudaDeviceProp prop;
  if ((e = cudaGetDeviceProperties(&prop, opt->device)) != cudaSuccess) return cuda_fail(e, "cudaGetDeviceProperties");
  // Kernel images exist only for sm_103a; setting attributes fails otherwise.
  if ((e = ipv::score_prepare(opt->max_frame_tokens, opt->max_head_dim)) != cudaSuccess)
    return cuda_fail(e, "no usable kernel image for this device (built for sm_103a)");
  if ((e = ipv::select_prepare(IPV_MAX_TOKENS)) != cudaSuccess) return cuda_fail(e, "select kernel set-up");
  if ((e = ipv::window_prepare()) != cudaSuccess) return cuda_fail(e, "fused kernel set-up");
  if ((e = ipv::pool_prepare()) != cudaSuccess) return cuda_fail(e, "pooling kernel set-up");
  State s;
  s.opt = *opt;
  s.num_sms = prop.multiProcessorCount;
  const size_t score_bytes = static_cast<size_t>(opt->max_slabs) * opt->token_capacity * sizeof(float);
  const size_t m_bytes =
      static_cast<size_t>(opt->max_slabs) * opt->max_frame_tokens * opt->max_head_dim * sizeof(float);
  const size_t flag_bytes = ipv::kWinFlags * static_cast<size_t>(opt->max_slabs) * sizeof(unsigned);
  if (cudaMalloc(&s.tar, score_bytes) != cudaSuccess || cudaMalloc(&s.van, score_bytes) != cudaSuccess ||
      cudaMalloc(&s.m, m_bytes) != cudaSuccess ||
      (opt->van_pool && cudaMalloc(&s.pooled, score_bytes) != cudaSuccess) ||
      (opt->head_shared && (cudaMalloc(&s.kk, score_bytes) != cudaSuccess ||
                            cudaMalloc(&s.tar_l, score_bytes) != cudaSuccess ||
                            cudaMalloc(&s.van_l, score_bytes) != cudaSuccess)) ||
      cudaMalloc(&s.wstate, sizeof(ipv::WinState)) != cudaSuccess ||
      cudaMalloc(&s.wflags, flag_bytes) != cudaSuccess || cudaMalloc(&s.claim, 3 * sizeof(unsigned)) != cudaSuccess) {
    cudaGetLastError();
    free_scratch(s);
    return fail(IPV_ENOMEM, "scratch of %zu bytes could not be allocated",
                (2 + opt->van_pool + 3 * opt->head_shared) * score_bytes + m_bytes);
  }
  if ((e = cudaMemset(s.wstate, 0, sizeof(ipv::WinState))) != cudaSuccess ||
      (e = cudaMemset(s.wflags, 0, flag_bytes)) != cudaSuccess ||
      (e = cudaMemset(s.claim, 0, 3 * sizeof(unsigned))) != cudaSuccess) {
    free_scratch(s);
    return cuda_fail(e, "clearing the fused pass's counters");
  }
  s.ready = true;
  g = s;
  g_err.clear();
  return IPV_OK;
}

int ipv_recent_frames(int64_t n_frames) {
  if (!g.ready || n_frames <= 0) return -1;
  return default_recent_frames(n_frames);
}

ipv_status ipv_score(const ipv_kv* k, const ipv_kv* v, int n_layers, int n_kv_heads, int head_dim,
                     int64_t n_tokens, int frame_grid_h, int frame_grid_w, float* tar_out,
                     float* van_out, void* stream) {
  Shape sh;
  if (!tar_out || !van_out) return fail(IPV_EINVAL, "tar_out and van_out must not be NULL");
  if ((reinterpret_cast<uintptr_t>(tar_out) & 3u) || (reinterpret_cast<uintptr_t>(van_out) & 3u))
    return fail(IPV_EINVAL, "score outputs must be 4-byte aligned");
  ipv_status s = check_cache(k, v, n_layers, n_kv_heads, head_dim, n_tokens, frame_grid_h,
                             frame_grid_w, false, &sh);
  if (s != IPV_OK) return s;
  if (sh.rp >= sh.N)
    return fail(IPV_EINVAL, "the %d recent frames leave no past tokens to score", sh.r);
  cudaSetDevice(g.opt.device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  ipv::ScoreArgs a{};
  a.k = k->buf[k->cur];
  a.v = v->buf[v->cur];
  a.patch_id = k->patch_id[k->cur];
  a.n_slabs = sh.S;
  a.cap = g.opt.token_capacity;
  a.n_tokens = sh.N;
  a.D = sh.D;
  a.p = sh.p;
  a.r = sh.r;
  a.is_bf16 = g.opt.dtype == IPV_BF16;
  a.m = g.m;
  a.tar = tar_out;
  a.van = van_out;
  a.zero_recent = 1;
  a.van_recent = g.opt.van_pool;
  a.num_sms = g.num_sms;
  const bool tar_frame = g.opt.ablation == IPV_ABLATION_TAR_FRAME;
  if (tar_frame && k->patch_id[k->cur] && !k->frame_id[k->cur])
    return fail(IPV_EINVAL, "the frame-level TaR needs frame ids for a cache with patch ids");
  if (g.opt.head_shared) {  // per-layer scores [n_layers][n_tokens]
    if ((s = check_shared(n_kv_heads, head_dim)) != IPV_OK) return s;
    cudaError_t e = launch_shared_scores(a, n_kv_heads, tar_out, van_out, 1, st);
    if (e == cudaSuccess && tar_frame) e = launch_tar_frame(tar_out, k, n_layers, n_kv_heads, sh, st);
    return after_launch(e, "scoring kernels");
  }
  prof_begin(0, st);
  cudaError_t e = ipv::launch_recent_mean(a, st);
  prof_end(0, st);
  if (e != cudaSuccess) return cuda_fail(e, "recent-frame mean kernel");
  prof_begin(1, st);
  e = ipv::launch_score(a, st);
  prof_end(1, st);
  if (e == cudaSuccess && tar_frame) e = launch_tar_frame(tar_out, k, sh.S, 1, sh, st);
  return after_launch(e, "scoring kernel");
}

ipv_status ipv_select(const float* tar, const float* van, int64_t n_slabs, int64_t n_tokens,
                      int frame_grid_h, int frame_grid_w, int64_t budget, float tar_ratio,
                      int32_t* kept_idx_out, void* stream) {
  if (!tar || !van) return fail(IPV_EINVAL, "score inputs must not be NULL");
  if (n_slabs <= 0 || n_tokens <= 0 || frame_grid_h <= 0 || frame_grid_w <= 0)
    return fail(IPV_EINVAL, "sizes must be positive");
  ipv_status s = check_select_args(n_tokens, budget, tar_ratio, kept_idx_out);
  if (s != IPV_OK) return s;
  const int64_t p = static_cast<int64_t>(frame_grid_h) * frame_grid_w;
  if (n_tokens % p != 0) return fail(IPV_EINVAL, "n_tokens is not a multiple of the frame size");
  if (n_slabs > INT32_MAX) return fail(IPV_EINVAL, "too many slabs");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  cudaSetDevice(g.opt.device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  if (n_tokens <= budget)
    return after_launch(ipv::launch_passthrough(kept_idx_out, n_slabs, n_tokens, budget, st),
                        "pass-through kernel");
  if (n_tokens > IPV_MAX_TOKENS) return fail(IPV_EINVAL, "n_tokens exceeds IPV_MAX_TOKENS");
  if (g.opt.ablation == IPV_ABLATION_UNIFORM) {  // whole frames at regular intervals; no score read
    if (budget % p != 0) return fail(IPV_EINVAL, "Uniform Select needs a budget of whole frames");
    prof_begin(2, st);
    cudaError_t e = ipv::launch_uniform(kept_idx_out, n_slabs, n_tokens, static_cast<int>(p), budget, st);
    prof_end(2, st);
    return after_launch(e, "uniform selection kernel");
  }
  const int64_t rp = static_cast<int64_t>(default_recent_frames(n_tokens / p)) * p;
  if (rp >= budget) return fail(IPV_EINVAL, "recent tokens r*p = %lld must be below budget", static_cast<long long>(rp));
  ipv::SelectArgs a{};
  a.tar = tar;
  a.van = van;
  a.n_slabs = n_slabs;
  a.n_tokens = n_tokens;
  a.rp = rp;
  a.budget = budget;
  split_budget(budget, tar_ratio, rp, &a.n_tar, &a.n_van);
  a.kept = kept_idx_out;
  a.num_sms = g.num_sms;
  prof_begin(2, st);
  cudaError_t e = ipv::launch_select(a, st);
  prof_end(2, st);
  return after_launch(e, "selection kernel");
}

ipv_status ipv_compress(ipv_kv* k, ipv_kv* v, int n_layers, int n_kv_heads, int head_dim,
                        int64_t n_tokens, int frame_grid_h, int frame_grid_w, int64_t budget,
                        float tar_ratio, int32_t* kept_idx_out, void* stream) {
  ipv_status s = check_select_args(n_tokens, budget, tar_ratio, kept_idx_out);
  if (s != IPV_OK) return s;
  Shape sh;
  s = check_cache(k, v, n_layers, n_kv_heads, head_dim, n_tokens, frame_grid_h, frame_grid_w,
                  n_tokens > budget, &sh);
  if (s != IPV_OK) return s;
  if (budget > g.opt.token_capacity)
    return fail(IPV_EINVAL, "budget %lld exceeds token_capacity %lld", static_cast<long long>(budget),
                static_cast<long long>(g.opt.token_capacity));
  cudaSetDevice(g.opt.device);
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const int64_t units = g.opt.head_shared ? n_layers : sh.S;  // rows of kept_idx_out
  if (g.opt.head_shared && (s = check_shared(n_kv_heads, head_dim)) != IPV_OK) return s;
  if (n_tokens <= budget)
    return after_launch(ipv::launch_passthrough(kept_idx_out, units, n_tokens, budget, st),
                        "pass-through kernel");
  if (n_tokens > IPV_MAX_TOKENS)
    return fail(IPV_EINVAL, "n_tokens %lld exceeds IPV_MAX_TOKENS", static_cast<long long>(n_tokens));
  const bool uniform = g.opt.ablation == IPV_ABLATION_UNIFORM;
  if (uniform && budget % sh.p != 0)
    return fail(IPV_EINVAL, "Uniform Select needs a budget of whole frames (budget %lld, p %d)",
                static_cast<long long>(budget), sh.p);
  if (!uniform && sh.rp >= budget)
    return fail(IPV_EINVAL, "recent tokens r*p = %lld must be below budget %lld", static_cast<long long>(sh.rp),
                static_cast<long long>(budget));
  if (g.opt.van_pool && k->patch_id[k->cur] && !k->frame_id[k->cur])
    return fail(IPV_EINVAL, "pooled VaN needs frame ids for a cache with patch ids");
  if (g.opt.van_pool && ipv::pool_smem_bytes(frame_grid_h, frame_grid_w, true) == 0)
    return fail(IPV_EINVAL, "frame too large for pooled VaN");
  if (g.opt.ablation == IPV_ABLATION_TAR_FRAME && k->patch_id[k->cur] && !k->frame_id[k->cur])
    return fail(IPV_EINVAL, "the frame-level TaR needs frame ids for a cache with patch ids");

  ipv::ScoreArgs a{};
  a.k = k->buf[k->cur];
  a.v = v->buf[v->cur];
  a.patch_id = k->patch_id[k->cur];
  a.n_slabs = sh.S;
  a.cap = g.opt.token_capacity;
  a.n_tokens = sh.N;
  a.D = sh.D;
  a.p = sh.p;
  a.r = sh.r;
  a.is_bf16 = g.opt.dtype == IPV_BF16;
  a.m = g.m;
  a.tar = g.tar;
  a.van = g.van;
  a.zero_recent = 0;
  a.van_recent = g.opt.van_pool;
  a.num_sms = g.num_sms;

  ipv::SelectArgs sa{};
  sa.tar = g.opt.head_shared ? g.tar_l : g.tar;
  sa.van = g.opt.van_pool ? g.pooled : g.opt.head_shared ? g.van_l : g.van;
  sa.n_slabs = units;
  sa.neg_tar = g.opt.ablation == IPV_ABLATION_TAR_REVERSE;
  sa.neg_van = g.opt.ablation == IPV_ABLATION_VAN_REVERSE;
  sa.n_tokens = sh.N;
  sa.rp = sh.rp;
  sa.budget = budget;
  split_budget(budget, tar_ratio, sh.rp, &sa.n_tar, &sa.n_van);
  sa.kept = kept_idx_out;
  sa.num_sms = g.num_sms;

  ipv::GatherArgs ga{};
  ga.k_src = k->buf[k->cur];
  ga.v_src = v->buf[v->cur];
  ga.k_dst = k->buf[1 - k->cur];
  ga.v_dst = v->buf[1 - v->cur];
  ga.pid_src = k->patch_id[k->cur];
  ga.pid_dst = k->patch_id[1 - k->cur];
  ga.fid_src = k->frame_id[k->cur];
  ga.fid_dst = k->frame_id[1 - k->cur];
  ga.kept = kept_idx_out;
  ga.n_slabs = sh.S;
  ga.cap = g.opt.token_capacity;
  ga.budget = budget;
  ga.row_bytes = sh.D * elem_bytes();
  ga.p = sh.p;
  ga.num_sms = g.num_sms;
  ga.heads_per_kept = g.opt.head_shared ? n_kv_heads : 1;
  ga.n_tokens = sh.N;
  ga.rp = sh.rp;
  ga.claim = g.claim;

  cudaError_t e;
  if (uniform) {  // no scores: the frames' rows, then all of them through the compaction
    prof_begin(2, st);
    e = ipv::launch_uniform(kept_idx_out, units, sh.N, sh.p, budget, st);
    prof_end(2, st);
    if (e != cudaSuccess) return cuda_fail(e, "uniform selection kernel");
    ga.rp = 0;
    prof_begin(3, st);
    e = ipv::launch_gather(ga, st);
    prof_end(3, st);
    if (e != cudaSuccess) return cuda_fail(e, "compaction kernel");
    k->cur = 1 - k->cur;
    v->cur = 1 - v->cur;
    return IPV_OK;
  }
  if (g.opt.single_kernel && !k->patch_id[k->cur]) {
    // The fused pass scores a cache that has never been compacted (row n is
    // patch n mod p); a cache with patch ids goes through the step kernels.
    ipv::WinArgs wa{};
    if (fused_args(a, sa, ga, sh, budget, &wa)) {
      if (g.win_dirty) {
        if ((e = cudaMemsetAsync(g.wstate, 0, offsetof(ipv::WinState, error), st)) != cudaSuccess ||
            (e = cudaMemsetAsync(g.wflags, 0, ipv::kWinFlags * sh.S * sizeof(unsigned), st)) != cudaSuccess)
          return cuda_fail(e, "clearing the fused pass's counters");
        g.win_dirty = false;
      }
      prof_begin(4, st);
      e = ipv::launch_window(wa, fused_smem(wa), st);
      prof_end(4, st);
      if (e != cudaSuccess) {
        g.win_dirty = true;
        return cuda_fail(e, "fused pass");
      }
      k->cur = 1 - k->cur;
      v->cur = 1 - v->cur;
      return IPV_OK;
    }
  }

  // Overlap: the compaction copies the recent rows (always kept) while the
  // latency-bound selection runs (see gather.cu).
  if (g.opt.head_shared) {
    e = launch_shared_scores(a, n_kv_heads, g.tar_l, g.van_l, 0, st);
    if (e != cudaSuccess) return cuda_fail(e, "scoring kernels");
  } else {
    prof_begin(0, st);
    e = ipv::launch_recent_mean(a, st);
    prof_end(0, st);
    if (e != cudaSuccess) return cuda_fail(e, "recent-frame mean kernel");
    prof_begin(1, st);
    e = ipv::launch_score(a, st);
    prof_end(1, st);
    if (e != cudaSuccess) return cuda_fail(e, "scoring kernel");
  }
  if (g.opt.ablation == IPV_ABLATION_TAR_FRAME) {
    e = launch_tar_frame(g.opt.head_shared ? g.tar_l : g.tar, k, units, g.opt.head_shared ? n_kv_heads : 1,
                         sh, st);
    if (e != cudaSuccess) return cuda_fail(e, "frame-level TaR kernel");
  }
  if (g.opt.van_pool) {  // the VaN stage ranks layer-adaptive pooled VaN
    // A layer is n_kv_heads slabs, or (shared index set) one unit whose ids
    // are those of its first head.
    const int hsh = g.opt.head_shared ? n_kv_heads : 1;
    ipv::PoolArgs pa{};
    pa.van = g.opt.head_shared ? g.van_l : g.van;
    pa.pooled = g.pooled;
    pa.patch_id = k->patch_id[k->cur];
    pa.frame_id = pa.patch_id ? k->frame_id[k->cur] : nullptr;
    pa.id_stride = g.opt.token_capacity * hsh;
    pa.n_slabs = units;
    pa.n_tokens = sh.N;
    pa.n_rows = sh.N - sh.rp;
    pa.n_heads = g.opt.head_shared ? 1 : n_kv_heads;
    pa.grid_h = frame_grid_h;
    pa.grid_w = frame_grid_w;
    for (int i = 0; i < 3; ++i) pa.tau[i] = g.opt.cv_tau[i];
    prof_begin(5, st);
    e = ipv::launch_pool(pa, st, true);
    prof_end(5, st);
    if (e != cudaSuccess) return cuda_fail(e, "VaN pooling kernel");
  }
  prof_begin(2, st);
  e = ipv::launch_select(sa, st);
  prof_end(2, st);
  if (e != cudaSuccess) return cuda_fail(e, "selection kernel");

  prof_begin(3, st);
  e = ipv::launch_gather(ga, st);
  prof_end(3, st);
  if (e != cudaSuccess) return cuda_fail(e, "compaction kernel");
  k->cur = 1 - k->cur;
  v->cur = 1 - v->cur;
  return IPV_OK;
}

ipv_status ipv_van_pool(const float* van, const uint16_t* patch_id, const uint32_t* frame_id,
                        int64_t id_stride, int n_layers, int n_kv_heads, int64_t n_tokens,
                        int frame_grid_h, int frame_grid_w, const float cv_tau[3],
                        float* pooled_out, int32_t* pool_size_out, void* stream) {
  if (!van || !pooled_out || !cv_tau) return fail(IPV_EINVAL, "van, pooled_out and cv_tau must not be NULL");
  if ((reinterpret_cast<uintptr_t>(van) & 3u) || (reinterpret_cast<uintptr_t>(pooled_out) & 3u) ||
      (reinterpret_cast<uintptr_t>(pool_size_out) & 3u) || (reinterpret_cast<uintptr_t>(frame_id) & 3u) ||
      (reinterpret_cast<uintptr_t>(patch_id) & 1u))
    return fail(IPV_EINVAL, "misaligned pointer");
  if (n_layers <= 0 || n_kv_heads <= 0 || n_tokens <= 0 || frame_grid_h <= 0 || frame_grid_w <= 0)
    return fail(IPV_EINVAL, "sizes must be positive");
  if (n_tokens > IPV_MAX_TOKENS) return fail(IPV_EINVAL, "n_tokens exceeds IPV_MAX_TOKENS");
  const int64_t p = static_cast<int64_t>(frame_grid_h) * frame_grid_w;
  if (p > IPV_MAX_POOL_FRAME_TOKENS)
    return fail(IPV_EINVAL, "frame of %lld tokens exceeds IPV_MAX_POOL_FRAME_TOKENS", static_cast<long long>(p));
  if (ipv::pool_smem_bytes(frame_grid_h, frame_grid_w, true) == 0) return fail(IPV_EINVAL, "frame too large for pooled VaN");
  if ((patch_id == nullptr) != (frame_id == nullptr))
    return fail(IPV_EINVAL, "patch_id and frame_id must both be set or both be NULL");
  if (patch_id && id_stride < n_tokens) return fail(IPV_EINVAL, "id_stride is below n_tokens");
  const float* t = cv_tau;
  if (t[0] != t[0] || t[1] != t[1] || t[2] != t[2] || !(t[0] <= t[1] && t[1] <= t[2]))
    return fail(IPV_EINVAL, "cv_tau must be ordered tau_1 <= tau_2 <= tau_3 (no NaN)");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  cudaSetDevice(g.opt.device);
  ipv::PoolArgs pa{};
  pa.van = van;
  pa.pooled = pooled_out;
  pa.pool_size = pool_size_out;
  pa.patch_id = patch_id;
  pa.frame_id = frame_id;
  pa.id_stride = id_stride;
  pa.n_slabs = static_cast<int64_t>(n_layers) * n_kv_heads;
  pa.n_tokens = n_tokens;
  pa.n_rows = n_tokens;
  pa.n_heads = n_kv_heads;
  pa.grid_h = frame_grid_h;
  pa.grid_w = frame_grid_w;
  for (int i = 0; i < 3; ++i) pa.tau[i] = t[i];
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  prof_begin(5, st);
  cudaError_t e = ipv::launch_pool(pa, st, false);
  prof_end(5, st);
  return after_launch(e, "VaN pooling kernel");
}

ipv_status ipv_append_frames(ipv_kv* k, ipv_kv* v, const void* k_new, const void* v_new, int n_layers,
                             int n_kv_heads, int head_dim, int64_t row0, int n_new_frames,
                             int frame_grid_h, int frame_grid_w, uint32_t first_frame, void* stream) {
  if (!k || !v || !k_new || !v_new) return fail(IPV_EINVAL, "k, v, k_new and v_new must not be NULL");
  if ((k->cur != 0 && k->cur != 1) || (v->cur != 0 && v->cur != 1)) return fail(IPV_EINVAL, "cur must be 0 or 1");
  if (n_layers <= 0 || n_kv_heads <= 0 || head_dim <= 0 || n_new_frames <= 0 || frame_grid_h <= 0 ||
      frame_grid_w <= 0 || row0 < 0)
    return fail(IPV_EINVAL, "sizes must be positive and row0 >= 0");
  const int64_t p = static_cast<int64_t>(frame_grid_h) * frame_grid_w;
  if (p > 65535) return fail(IPV_EINVAL, "frame_grid_h*frame_grid_w exceeds 65535");
  void* kd = k->buf[k->cur];
  void* vd = v->buf[v->cur];
  if (!kd || !vd || kd == vd) return fail(IPV_EINVAL, "live halves must be distinct and not NULL");
  if (!aligned16(kd) || !aligned16(vd) || !aligned16(k_new) || !aligned16(v_new))
    return fail(IPV_EINVAL, "cache halves and new rows must be 16-byte aligned");
  const uint32_t* fid = k->frame_id[k->cur];
  if (fid && (reinterpret_cast<uintptr_t>(fid) & 3u)) return fail(IPV_EINVAL, "frame ids must be 4-byte aligned");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  const int64_t S = static_cast<int64_t>(n_layers) * n_kv_heads;
  const int64_t n_new = static_cast<int64_t>(n_new_frames) * p;
  if (S > g.opt.max_slabs) return fail(IPV_EINVAL, "n_layers*n_kv_heads exceeds max_slabs");
  if (head_dim > g.opt.max_head_dim) return fail(IPV_EINVAL, "head_dim exceeds max_head_dim");
  if ((static_cast<int64_t>(head_dim) * elem_bytes()) % 16 != 0)
    return fail(IPV_EINVAL, "head_dim*element size must be a multiple of 16 bytes");
  if (row0 + n_new > g.opt.token_capacity)
    return fail(IPV_EINVAL, "row0 + %lld new rows exceed token_capacity %lld", static_cast<long long>(n_new),
                static_cast<long long>(g.opt.token_capacity));
  cudaSetDevice(g.opt.device);
  ipv::AppendArgs a{};
  a.k_new = k_new;
  a.v_new = v_new;
  a.k_dst = kd;
  a.v_dst = vd;
  a.pid = k->patch_id[k->cur];
  a.fid = k->frame_id[k->cur];
  a.n_slabs = S;
  a.cap = g.opt.token_capacity;
  a.row0 = row0;
  a.n_new = n_new;
  a.row_bytes = head_dim * elem_bytes();
  a.p = static_cast<int>(p);
  a.first_frame = first_frame;
  a.num_sms = g.num_sms;
  return after_launch(ipv::launch_append(a, static_cast<cudaStream_t>(stream)), "append kernel");
}

ipv_status ipv_set_wait_limit(int64_t polls) {
  if (polls < 0) return fail(IPV_EINVAL, "polls must be >= 0");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  g.wait_limit = polls > 0 ? polls : int64_t{1} << 20;
  return IPV_OK;
}

ipv_status ipv_device_error(uint32_t* err_out) {
  if (!err_out) return fail(IPV_EINVAL, "err_out must not be NULL");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  cudaSetDevice(g.opt.device);
  cudaError_t e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_fail(e, "cudaDeviceSynchronize");
  ipv::WinState ws;
  if ((e = cudaMemcpy(&ws, g.wstate, sizeof ws, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "reading the fused pass's state");
  *err_out = ws.error;
  if (ws.error != 0u) {
    ws.error = 0u;
    if ((e = cudaMemcpy(g.wstate, &ws, sizeof ws, cudaMemcpyHostToDevice)) != cudaSuccess)
      return cuda_fail(e, "clearing the fused pass's error word");
  }
  return IPV_OK;
}

ipv_status ipv_profile_enable(int on) {
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  cudaSetDevice(g.opt.device);
  // Create the events up front so that timed loops do not pay for it.
  while (on && g.pool.size() < 4096) {
    EventPair p;
    if (cudaEventCreate(&p.start) != cudaSuccess || cudaEventCreate(&p.stop) != cudaSuccess)
      return cuda_fail(cudaGetLastError(), "cudaEventCreate");
    g.pool.push_back(p);
  }
  g.profiling = on != 0;
  return IPV_OK;
}

ipv_status ipv_profile_collect(double ms_out[IPV_NUM_KERNELS], int64_t launches_out[IPV_NUM_KERNELS],
                               int timeout_ms) {
  if (!ms_out || !launches_out) return fail(IPV_EINVAL, "outputs must not be NULL");
  if (!g.ready) return fail(IPV_ENOINIT, "ipv_init has not succeeded");
  cudaSetDevice(g.opt.device);
  for (int id = 0; id < IPV_NUM_KERNELS; ++id) {
    ms_out[id] = 0.0;
    launches_out[id] = 0;
  }
  // Bounded wait for the last recorded stop event of every kernel id.
  const int step_us = 200;
  int waited_us = 0;
  for (int id = 0; id < IPV_NUM_KERNELS; ++id) {
    if (g.pending[id].empty()) continue;
    for (;;) {
      cudaError_t q = cudaEventQuery(g.pending[id].back().stop);
      if (q == cudaSuccess) break;
      if (q != cudaErrorNotReady) return cuda_fail(q, "cudaEventQuery");
      if (waited_us >= timeout_ms * 1000) return fail(IPV_ETIMEOUT, "profiling events not complete after %d ms", timeout_ms);
      struct timespec ts = {0, step_us * 1000};
      nanosleep(&ts, nullptr);
      waited_us += step_us;
    }
  }
  for (int id = 0; id < IPV_NUM_KERNELS; ++id) {
    for (auto& p : g.pending[id]) {
      float ms = 0.0f;
      cudaError_t e = cudaEventElapsedTime(&ms, p.start, p.stop);
      if (e != cudaSuccess) return cuda_fail(e, "cudaEventElapsedTime");
      ms_out[id] += ms;
      launches_out[id] += 1;
      g.pool.push_back(p);
    }
    g.pending[id].clear();
  }
  return IPV_OK;
}

}  // extern "C"
