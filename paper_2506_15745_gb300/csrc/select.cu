// Step (iii) of the compression pass: the split-budget selection, a
// 1024-thread block per (layer, KV head) slab (for larger slabs, one block per
// SM taking slabs in turn). The algorithm (Sec. 3.3; Algorithm 1 steps 3-5)
// is dev::select_slab_reg in pass_device.cuh (keys in registers), or
// dev::select_slab (keys in shared memory) for larger slabs.
#include "pass_device.cuh"

namespace ipv {
namespace {

#ifndef IPV_SELECT_MAXNREG
#define IPV_SELECT_MAXNREG 48
#endif

// Slabs blockIdx.x, blockIdx.x + gridDim.x, ...: with one block per SM the
// whole grid starts at once, so the compaction (launched when every block of
// this grid has started) puts a block beside each of them and copies the
// recent rows while the selection runs, as it does beside the register
// kernel. 48 registers leave it room (1024 x 48 + 256 x 64 = 65,536).
__global__ void __maxnreg__(IPV_SELECT_MAXNREG) select_kernel(SelectArgs a) {
  extern __shared__ __align__(16) uint32_t sm_sel[];
  __shared__ dev::SelShared sh;
  pdl_trigger();
  pdl_wait();  // the scores come from the scoring kernel
  for (int64_t s = blockIdx.x; s < a.n_slabs; s += gridDim.x) dev::select_slab<kSelectThreads>(a, s, sm_sel, sh);
}

// The same selection with every thread's share of the scores in registers
// (at most E past tokens per thread). Its shared memory is cleared before it
// waits for the scoring kernel. 48 registers per thread leave room for one
// compaction block beside each selection block (1024 x 48 + 256 x 64 =
// 65,536), which copies the recent rows while the selection runs: a few
// spills cost less than the copy bandwidth a full register file would
// shut out (LLaVA-OV-7B shape: pass 0.2120 against 0.2155 ms at 64).
template <int E>
__global__ void __maxnreg__(IPV_SELECT_MAXNREG) select_reg_kernel(SelectArgs a) {
  extern __shared__ __align__(16) uint32_t sm_sel[];
  __shared__ dev::SelShared sh;
  pdl_trigger();
  dev::select_reg_clear<kSelectThreads, E>(sm_sel, sh);
  pdl_wait();  // the scores come from the scoring kernel
  dev::select_slab_reg<kSelectThreads, E, true>(a, blockIdx.x, sm_sel, sh);
}
#ifndef IPV_SELECT_REG_SMALL_E
#define IPV_SELECT_REG_SMALL_E 9
#endif
constexpr int kSelectRegSmallE = IPV_SELECT_REG_SMALL_E;  // fewer registers when a slab needs no more

template <int E>
constexpr size_t reg_smem_bytes() {
  return dev::select_reg_smem_words<kSelectThreads, E>() * sizeof(uint32_t);
}

// The index rows of the index kernels below are the same for every slab:
// block (x, y) computes columns j = x 256 + t, ... once and stores them to
// rows y, y + gridDim.y, ... (coalesced along j, no division per element).
constexpr int kIndexThreads = 256;
constexpr int64_t kIndexRowBlocks = 32;

__global__ void passthrough_kernel(int32_t* kept, int64_t n_slabs, int64_t n_tokens,
                                   int64_t budget) {
  for (int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; j < budget;
       j += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int32_t v = j < n_tokens ? static_cast<int32_t>(j) : -1;
    for (int64_t row = blockIdx.y; row < n_slabs; row += gridDim.y) kept[row * budget + j] = v;
  }
}

// Uniform Select (Sec. 4 ablation table; frames at regular intervals, all
// their tokens kept): element j of a unit's kept row is row q of the a-th
// kept frame in ascending order, a = j div p, q = j mod p, whose frame is
// F - 1 - floor((k - 1 - a) F / k). No score is read.
__global__ void uniform_kernel(int32_t* kept, int64_t units, int64_t n_frames, int p, int64_t k) {
  pdl_trigger();
  const int64_t per = k * p;
  for (int64_t j = blockIdx.x * static_cast<int64_t>(blockDim.x) + threadIdx.x; j < per;
       j += static_cast<int64_t>(gridDim.x) * blockDim.x) {
    const int64_t a = j / p;
    const int64_t f = n_frames - 1 - ((k - 1 - a) * n_frames) / k;
    const int32_t v = static_cast<int32_t>(f * p + (j - a * p));
    for (int64_t row = blockIdx.y; row < units; row += gridDim.y) kept[row * per + j] = v;
  }
}

dim3 index_grid(int64_t rows, int64_t cols) {
  const int64_t bx = (cols + kIndexThreads - 1) / kIndexThreads;
  return dim3(static_cast<unsigned>(bx < 4096 ? bx : 4096),
              static_cast<unsigned>(rows < kIndexRowBlocks ? rows : kIndexRowBlocks));
}

}  // namespace

cudaError_t launch_uniform(int32_t* kept, int64_t units, int64_t n_tokens, int p, int64_t budget,
                           cudaStream_t st) {
  uniform_kernel<<<index_grid(units, budget), kIndexThreads, 0, st>>>(kept, units, n_tokens / p, p, budget / p);
  return cudaGetLastError();
}

size_t select_smem_bytes(int64_t n_past) {
  return dev::select_smem_words<kSelectThreads>(n_past) * sizeof(uint32_t);
}

namespace {
// VaN in shared memory too while that stays within what select_prepare allows.
bool van_fits(int64_t n_past) {
  return dev::select_smem_words<kSelectThreads>(n_past, true) <=
         dev::select_smem_words<kSelectThreads>(kMaxTokens);
}
}  // namespace

cudaError_t select_prepare(int64_t max_tokens) {
  cudaError_t e = cudaFuncSetAttribute(select_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                       static_cast<int>(select_smem_bytes(max_tokens)));
  if (e != cudaSuccess) return e;
  e = cudaFuncSetAttribute(select_reg_kernel<kSelectRegSmallE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(reg_smem_bytes<kSelectRegSmallE>()));
  if (e != cudaSuccess) return e;
  return cudaFuncSetAttribute(select_reg_kernel<kSelectRegE>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                              static_cast<int>(reg_smem_bytes<kSelectRegE>()));
}

cudaError_t launch_select(const SelectArgs& a, cudaStream_t st) {
  SelectArgs b = a;
  const int64_t n_past = a.n_tokens - a.rp;
  if (n_past <= static_cast<int64_t>(kSelectThreads) * kSelectRegE) {
    if (n_past <= static_cast<int64_t>(kSelectThreads) * kSelectRegSmallE)
      return launch(select_reg_kernel<kSelectRegSmallE>, static_cast<unsigned>(a.n_slabs), kSelectThreads,
                    reg_smem_bytes<kSelectRegSmallE>(), st, true, b);
    return launch(select_reg_kernel<kSelectRegE>, static_cast<unsigned>(a.n_slabs), kSelectThreads,
                  reg_smem_bytes<kSelectRegE>(), st, true, b);
  }
  b.van_smem = van_fits(n_past) ? 1 : 0;
  const size_t smem = dev::select_smem_words<kSelectThreads>(n_past, b.van_smem != 0) * sizeof(uint32_t);
  const int64_t grid = a.num_sms > 0 && a.num_sms < a.n_slabs ? a.num_sms : a.n_slabs;
  return launch(select_kernel, static_cast<unsigned>(grid), kSelectThreads, smem, st, true, b);
}

cudaError_t launch_passthrough(int32_t* kept, int64_t n_slabs, int64_t n_tokens, int64_t budget,
                               cudaStream_t st) {
  passthrough_kernel<<<index_grid(n_slabs, budget), kIndexThreads, 0, st>>>(kept, n_slabs, n_tokens, budget);
  return cudaGetLastError();
}

}  // namespace ipv
