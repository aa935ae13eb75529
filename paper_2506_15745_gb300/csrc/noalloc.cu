// ipv_compress_static: the compression pass without any device allocation.
//
// ipv_compress keeps its per-call working memory (the TaR and VaN score of
// every token and the recent-frame mean of every patch) in buffers that
// ipv_init obtains with cudaMalloc. Some callers cannot allocate device memory
// at all: a process whose device memory is owned by a caching allocator or a
// fixed budget that the library must not grow (a memory-capped streaming
// server is exactly that), or code on a latency-critical path where cudaMalloc
// and cudaFree, which can synchronise the device, are not allowed. This entry
// point serves them: it runs the same kernels as ipv_compress, but its working
// memory is one statically sized array in this library's device image,
// reserved when the library's code is loaded on a device and held until the
// process exits. It needs no ipv_init.
//
// On the first call on a device (the current device), the entry point sets
// up that device once: it sets the kernels' shared-memory limits and looks up
// the array's device address with cudaGetSymbolAddress. Make that first call
// before any stream capture. The set-up is kept for the life of the process:
// a cudaDeviceReset of that device after its first call is not supported.
// All calls on a device share the one array, which
// keeps whatever the previous call left: calls that may overlap on the GPU
// (different streams, or different host threads) race on it and must be
// ordered by the caller. Nothing in the array needs clearing between calls,
// because every word a call reads was written earlier in that same call.
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <mutex>

#include "ipv.h"
#include "ipv_common.cuh"

namespace ipv {
void record_error(ipv_status s, const char* msg);
}

namespace {

static_assert(IPV_STATIC_SCRATCH_BYTES % 256 == 0, "scratch size");

// The working memory of every ipv_compress_static call on this device.
static __device__ __align__(256) unsigned char g_static_scratch[IPV_STATIC_SCRATCH_BYTES];
// The compaction's work counters (zero between passes).
static __device__ unsigned g_static_claim[3];

struct DeviceSetup {
  bool done = false;
  unsigned char* scratch = nullptr;  // device address of g_static_scratch
  unsigned* claim = nullptr;         // device address of g_static_claim
  int num_sms = 0;
};

constexpr int kMaxDevices = 64;
DeviceSetup g_setup[kMaxDevices];
std::mutex g_setup_mu;

ipv_status reject(ipv_status s, const char* fmt, ...) {
  char buf[512];
  va_list ap;
  va_start(ap, fmt);
  std::vsnprintf(buf, sizeof buf, fmt, ap);
  va_end(ap);
  ipv::record_error(s, buf);
  return s;
}

ipv_status cuda_reject(cudaError_t e, const char* what) {
  return reject(IPV_ECUDA, "%s: %s (%s)", what, cudaGetErrorName(e), cudaGetErrorString(e));
}

// Once per device, with that device current: kernel limits, the array's address.
ipv_status setup_current_device(DeviceSetup** out) {
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_reject(e, "cudaGetDevice");
  if (dev < 0 || dev >= kMaxDevices) return reject(IPV_EINVAL, "device ordinal %d not supported", dev);
  std::lock_guard<std::mutex> lock(g_setup_mu);
  DeviceSetup& d = g_setup[dev];
  if (!d.done) {
    if ((e = ipv::score_prepare(0, 0)) != cudaSuccess)
      return cuda_reject(e, "no usable kernel image for this device (built for sm_103a)");
    if ((e = ipv::select_prepare(IPV_MAX_TOKENS)) != cudaSuccess) return cuda_reject(e, "select kernel set-up");
    void* ptr = nullptr;
    if ((e = cudaGetSymbolAddress(&ptr, g_static_scratch)) != cudaSuccess)
      return cuda_reject(e, "cudaGetSymbolAddress of the static scratch");
    void* cptr = nullptr;
    if ((e = cudaGetSymbolAddress(&cptr, g_static_claim)) != cudaSuccess)
      return cuda_reject(e, "cudaGetSymbolAddress of the compaction counters");
    d.claim = static_cast<unsigned*>(cptr);
    if ((e = cudaDeviceGetAttribute(&d.num_sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess)
      return cuda_reject(e, "cudaDeviceGetAttribute");
    d.scratch = static_cast<unsigned char*>(ptr);
    d.done = true;
  }
  *out = &d;
  return IPV_OK;
}

size_t round256(size_t b) { return (b + 255) & ~static_cast<size_t>(255); }

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }

}  // namespace

extern "C" ipv_status ipv_compress_static(ipv_kv* k, ipv_kv* v, ipv_dtype dtype, int64_t token_capacity,
                                          int recent_frames, int n_layers, int n_kv_heads, int head_dim,
                                          int64_t n_tokens, int frame_grid_h, int frame_grid_w,
                                          int64_t budget, float tar_ratio, int32_t* kept_idx_out,
                                          void* stream) {
  // The argument rules of ipv_compress, with the options of ipv_init as arguments.
  if (!k || !v || !kept_idx_out) return reject(IPV_EINVAL, "k, v and kept_idx_out must not be NULL");
  if (dtype != IPV_BF16 && dtype != IPV_F32) return reject(IPV_EINVAL, "unknown dtype %d", dtype);
  if (k->cur != 0 && k->cur != 1) return reject(IPV_EINVAL, "k->cur must be 0 or 1");
  if (v->cur != 0 && v->cur != 1) return reject(IPV_EINVAL, "v->cur must be 0 or 1");
  if (n_layers <= 0 || n_kv_heads <= 0 || head_dim <= 0 || n_tokens <= 0 || frame_grid_h <= 0 ||
      frame_grid_w <= 0 || budget <= 0 || token_capacity <= 0 || recent_frames < 0)
    return reject(IPV_EINVAL, "sizes must be positive (recent_frames >= 0)");
  if (head_dim > 512) return reject(IPV_EINVAL, "head_dim %d exceeds 512", head_dim);
  const int elem = dtype == IPV_BF16 ? 2 : 4;
  if ((head_dim * elem) % 16 != 0) return reject(IPV_EINVAL, "head_dim*element size must be a multiple of 16 bytes");
  const int64_t p = static_cast<int64_t>(frame_grid_h) * frame_grid_w;
  if (p > 65535) return reject(IPV_EINVAL, "frame_grid_h*frame_grid_w exceeds 65535");
  if (n_tokens % p != 0) return reject(IPV_EINVAL, "n_tokens is not a multiple of the frame size");
  if (n_tokens > token_capacity || budget > token_capacity || token_capacity > INT32_MAX)
    return reject(IPV_EINVAL, "n_tokens and budget must not exceed token_capacity (< 2^31)");
  if (!(tar_ratio >= 0.0f && tar_ratio <= 1.0f)) return reject(IPV_EINVAL, "tar_ratio must lie in [0, 1]");
  if (!aligned(kept_idx_out, 4)) return reject(IPV_EINVAL, "kept_idx_out must be 4-byte aligned");
  const bool evict = n_tokens > budget;
  void* ks = k->buf[k->cur];
  void* vs = v->buf[v->cur];
  void* kd = k->buf[1 - k->cur];
  void* vd = v->buf[1 - v->cur];
  if (!ks || !vs || !aligned(ks, 16) || !aligned(vs, 16) || ks == vs)
    return reject(IPV_EINVAL, "live cache halves must be distinct, non-NULL and 16-byte aligned");
  if (evict && (!kd || !vd || !aligned(kd, 16) || !aligned(vd, 16) || kd == ks || vd == vs || kd == vs ||
                vd == ks || kd == vd))
    return reject(IPV_EINVAL, "destination halves must be distinct, non-NULL and 16-byte aligned");
  const uint16_t* pid_src = k->patch_id[k->cur];
  uint16_t* pid_dst = k->patch_id[1 - k->cur];
  if (evict && pid_dst && pid_dst == pid_src) return reject(IPV_EINVAL, "patch-id halves must be distinct");
  if (evict && (!aligned(k->frame_id[0], 4) || !aligned(k->frame_id[1], 4) ||
                (k->frame_id[1 - k->cur] && k->frame_id[1 - k->cur] == k->frame_id[k->cur])))
    return reject(IPV_EINVAL, "frame-id halves must be distinct and 4-byte aligned");
  const int64_t S = static_cast<int64_t>(n_layers) * n_kv_heads;
  const int64_t f = n_tokens / p;
  int r = recent_frames;
  if (r == 0) {
    const int64_t rr = static_cast<int64_t>(std::floor(static_cast<double>(f) / 8.0 + 0.5));
    r = static_cast<int>(rr < 1 ? 1 : rr);
  }
  const int64_t rp = static_cast<int64_t>(r) * p;

  // Working memory: TaR and VaN [S][n_tokens], m [S][p][head_dim] (fp32).
  // The slab count is bounded by division first, so that the byte counts
  // below cannot wrap around for any argument values.
  if (S > INT32_MAX) return reject(IPV_EINVAL, "n_layers*n_kv_heads exceeds 2^31 - 1");
  const uint64_t per_slab = 8u * static_cast<uint64_t>(n_tokens) + 4u * static_cast<uint64_t>(p) * head_dim;
  if (evict && static_cast<uint64_t>(S) > IPV_STATIC_SCRATCH_BYTES / per_slab)
    return reject(IPV_EINVAL,
                  "this pass needs more than the %u bytes of working memory of ipv_compress_static "
                  "(%lld slabs of %llu bytes; use ipv_compress, or fewer slabs per call)",
                  static_cast<unsigned>(IPV_STATIC_SCRATCH_BYTES), static_cast<long long>(S),
                  static_cast<unsigned long long>(per_slab));
  const size_t score_bytes = round256(static_cast<size_t>(S) * n_tokens * sizeof(float));
  const size_t m_bytes = round256(static_cast<size_t>(S) * p * head_dim * sizeof(float));
  if (evict && 2 * score_bytes + m_bytes > IPV_STATIC_SCRATCH_BYTES)
    return reject(IPV_EINVAL,
                  "this pass needs %zu bytes of working memory; ipv_compress_static has %u "
                  "(use ipv_compress, or fewer slabs per call)",
                  2 * score_bytes + m_bytes, static_cast<unsigned>(IPV_STATIC_SCRATCH_BYTES));
  if (evict && n_tokens > IPV_MAX_TOKENS) return reject(IPV_EINVAL, "n_tokens exceeds IPV_MAX_TOKENS");
  if (evict && rp >= budget) return reject(IPV_EINVAL, "recent tokens r*p must be below budget");

  DeviceSetup* dev = nullptr;
  ipv_status st = setup_current_device(&dev);
  if (st != IPV_OK) return st;
  cudaStream_t cs = static_cast<cudaStream_t>(stream);
  cudaError_t e;
  if (!evict) {
    if ((e = ipv::launch_passthrough(kept_idx_out, S, n_tokens, budget, cs)) != cudaSuccess)
      return cuda_reject(e, "pass-through kernel");
    return IPV_OK;
  }

  float* tar = reinterpret_cast<float*>(dev->scratch);
  float* van = reinterpret_cast<float*>(dev->scratch + score_bytes);
  float* m = reinterpret_cast<float*>(dev->scratch + 2 * score_bytes);

  ipv::ScoreArgs a{};
  a.k = ks;
  a.v = vs;
  a.patch_id = pid_src;
  a.n_slabs = S;
  a.cap = token_capacity;
  a.n_tokens = n_tokens;
  a.D = head_dim;
  a.p = static_cast<int>(p);
  a.r = r;
  a.is_bf16 = dtype == IPV_BF16;
  a.m = m;
  a.tar = tar;
  a.van = van;
  a.zero_recent = 0;
  a.num_sms = dev->num_sms;
  if ((e = ipv::launch_recent_mean(a, cs)) != cudaSuccess) return cuda_reject(e, "recent-frame mean kernel");
  if ((e = ipv::launch_score(a, cs)) != cudaSuccess) return cuda_reject(e, "scoring kernel");

  ipv::SelectArgs sa{};
  sa.tar = tar;
  sa.van = van;
  sa.n_slabs = S;
  sa.n_tokens = n_tokens;
  sa.rp = rp;
  sa.budget = budget;
  // floor(alpha * budget) for TaR including the r p recent tokens, the rest for VaN.
  const int64_t share = static_cast<int64_t>(std::floor(static_cast<double>(tar_ratio) * budget));
  sa.n_tar = share > rp ? share - rp : 0;
  sa.n_van = budget - rp - sa.n_tar;
  sa.kept = kept_idx_out;
  sa.num_sms = dev->num_sms;
  if ((e = ipv::launch_select(sa, cs)) != cudaSuccess) return cuda_reject(e, "selection kernel");

  ipv::GatherArgs ga{};
  ga.k_src = ks;
  ga.v_src = vs;
  ga.k_dst = kd;
  ga.v_dst = vd;
  ga.pid_src = pid_src;
  ga.pid_dst = pid_dst;
  ga.fid_src = k->frame_id[k->cur];
  ga.fid_dst = k->frame_id[1 - k->cur];
  ga.kept = kept_idx_out;
  ga.n_slabs = S;
  ga.cap = token_capacity;
  ga.budget = budget;
  ga.row_bytes = head_dim * elem;
  ga.p = static_cast<int>(p);
  ga.num_sms = dev->num_sms;
  ga.n_tokens = n_tokens;
  ga.rp = rp;
  ga.claim = dev->claim;
  if ((e = ipv::launch_gather(ga, cs)) != cudaSuccess) return cuda_reject(e, "compaction kernel");
  k->cur = 1 - k->cur;
  v->cur = 1 - v->cur;
  return IPV_OK;
}
